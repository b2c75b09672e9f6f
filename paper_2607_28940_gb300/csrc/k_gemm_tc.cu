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




constexpr int kStageNAtt = 512;   // bias entries staged with the fused attention (N = d <= 512)
constexpr int kStageNSrv = 1536;  // bias entries staged with the fused serving attention (N = 3 d <= 1536)
constexpr int kSrvMaxS = 8;       // context rows per request the fused serving attention takes
constexpr int kSrvSlots = kSrvMaxS + 1;

// Fused LOCAL_GLOBAL cross-attention (EPI_ATTN_LG): each epilogue warp owns
// 64 query columns (one head of 64 or two of 32) of 32 rows.  Per request
// among its rows it stages the K/V columns its heads read as 16 key slots of
// bf16: slots 0 .. W-1 the window rows, W .. 14 zero, 15 the anchor.
constexpr int kAttKeys = 16;                  // key slots: window (at most 15 rows) + anchor
constexpr int kAttAnchor = kAttKeys - 1;
constexpr int kAttWinMax = kAttKeys - 1;      // longest window the fused path takes
constexpr int kAttCols = 64;                  // query columns per epilogue warp
constexpr int kAttKvBytes = kAttKeys * kAttCols * 2;   // one of K, V staged for one warp

constexpr int kEpiWarps = 8;                  // two warps per TMEM lane quarter
constexpr int NUM_THREADS = 64 + 32 * kEpiWarps;
constexpr int kRedStride = 17;                // per-row exchange slots: sum + 16 logits

// Epilogue of one 128 x BN tile for one warp: TMEM lanes `tlane` (32 rows of
// the tile), columns [c0, c0 + BN/2) of the accumulator.  The two warps that
// share a lane quarter exchange row sums (and head logits) through `red`.
template <int BN, int EPI, int NAP, int SB>
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
      store_chunk<SB>(vals, out, valid, tma_ok, tmO, tx, ty, stage, kchunk++, lane);
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
        store_chunk<SB>(v, out + c, valid, true, tmO, c0 + c, ty, stage, kchunk++, lane);
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

// ------------------------------------------------------------------ fused LOCAL_GLOBAL attention

// The attention of one warp's 32 query rows against one request's 16 key
// slots is two small matrix products per head, S = Q K^T (32 x 16, inner
// dimension d_h) and O = P V (32 x d_h, inner dimension 16).  They run as
// warp-level bf16 MMAs (m16n8k16, fp32 accumulation) on shared-memory tiles
// of this warp; the softmax runs on the S fragments in registers, and the P
// fragments are the A operand of the second product (the S accumulator
// layout of two 8-key tiles is the A layout of one 16-key step).  The
// tcgen05 MMAs of the projection are issued by one thread for the whole
// 128-row tile; these products belong to each warp's own rows and keys.

__device__ __forceinline__ void mma_16816(float* d, const uint32_t* a, const uint32_t* b) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
      "{%0,%1,%2,%3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b[0]), "r"(b[1]));
}
__device__ __forceinline__ void ldsm_x4(uint32_t* r, uint32_t addr) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(addr));
}
__device__ __forceinline__ void ldsm_x4_t(uint32_t* r, uint32_t addr) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(addr));
}
__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
  __nv_bfloat162 h = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&h);
}
// Byte offset of 16-byte unit u of row r in a [rows][64] bf16 tile (128-byte
// rows; units XOR-swizzled by the row so that eight rows read as an 8 x 8
// matrix hit distinct banks).
__device__ __forceinline__ uint32_t tile_off(int r, int u) {
  return static_cast<uint32_t>(r * 128 + ((u ^ (r & 7)) << 4));
}

// Row tile of tile t in the fused-attention kernel: the row tiles are
// rotated so that the last one (the context-token rows of every request,
// whose warps attend to many requests each) is processed in the first round
// by the last CTAs (or pairs: `slots` tiles run at once), which have no
// extra tile in the last round.
__device__ __forceinline__ int att_tile_m(int t, int n_tiles, int m_tiles, int slots) {
  const int shift = slots / n_tiles - 1;   // first-round position of the last row tile
  return (t / n_tiles + m_tiles - 1 + (m_tiles - shift % m_tiles)) % m_tiles;
}

__device__ __forceinline__ void cp_async16(uint32_t dst, const void* src, uint32_t src_bytes) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(dst), "l"(src), "r"(src_bytes) : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
__device__ __forceinline__ void cp_async_wait_all() { asm volatile("cp.async.wait_all;" ::: "memory"); }

// Shared memory of one epilogue warp for the fused attention: two K/V
// buffers (16 key slots x 64 columns bf16 each for K and V) and two fp32
// anchor rows (K then V, 64 columns each); q and the outputs use the warp's
// bulk-store staging buffers.
constexpr int kAttBufBytes = 2 * kAttKvBytes + 2 * kAttCols * 4;
constexpr int kAttWarpBytes = 2 * kAttBufBytes;

// This lane's row: its request, that request's window rows and first window
// row in the cache (W = 0 for a row past M).
struct AttRow {
  int r;
  int W;
  long long base;
};
__device__ __forceinline__ void att_row_meta(const EpiArgs& e, AttRow& a) {
  a.W = 0;
  a.base = 0;
  if (a.r >= 0) {
    const int len = __ldg(e.att_kv_len + a.r);
    const int lo = len > e.att_l_local ? len - e.att_l_local : 0;
    a.W = len - lo;                                           // <= kAttWinMax (checked on the host)
    a.base = static_cast<long long>(__ldg(e.att_kv_off + a.r)) + lo;
  }
}

// K/V columns [kc0, kc0 + kvw) read by the heads of query columns
// [col0, col0 + 64): kvw is 32 or 64, a whole number of heads (d_h = 32 or
// 64, so the head index is a shift).
__device__ __forceinline__ void att_kv_cols(const EpiArgs& e, int col0, int& kc0, int& kvw) {
  const int lg = e.att_dh == 64 ? 6 : 5, grp = e.att_group;
  const int h0 = col0 >> lg, h1 = (col0 + kAttCols - 1) >> lg;
  const int g0 = grp == 1 ? h0 : h0 / grp, g1 = grp == 1 ? h1 : h1 / grp;
  kc0 = g0 << lg;
  kvw = ((g1 - g0) << lg) + e.att_dh;
}

// Starts the asynchronous copies of request rc's key slots into buffer `buf`:
// window rows 0 .. W-1 of the K and V columns [kc0, kc0 + kvw), zero-filled
// slots W .. 14, and the fp32 anchor columns; one commit group.
__device__ __forceinline__ void att_issue(const EpiArgs& e, int rc, int W, long long base, int kc0, int kvw,
                                          uint8_t* buf, int lane) {
  const __nv_bfloat16* Kc = static_cast<const __nv_bfloat16*>(e.att_k);
  const __nv_bfloat16* Vc = static_cast<const __nv_bfloat16*>(e.att_v);
  const uint32_t sK = smem_u32(buf), sV = sK + kAttKvBytes, sA = sV + kAttKvBytes;
  const int sh = kvw == 64 ? 3 : 2;                        // 16-byte units per row: 8 or 4
  const long long dkv = e.att_dkv;
  for (int idx = lane; idx < (kAttWinMax << sh); idx += 32) {
    const int t = idx >> sh, u = idx & ((1 << sh) - 1);
    const bool in = t < W;
    const long long src = (base + (in ? t : 0)) * dkv + kc0 + 8 * u;   // a valid row when zero-filling
    cp_async16(sK + tile_off(t, u), Kc + src, in ? 16u : 0u);
    cp_async16(sV + tile_off(t, u), Vc + src, in ? 16u : 0u);
  }
  const int q4 = kvw / 4;
  for (int i = lane; i < 2 * q4; i += 32) {
    const bool isv = i >= q4;
    const int c = 4 * (isv ? i - q4 : i);
    cp_async16(sA + (isv ? kAttCols * 4 : 0) + 4 * c, (isv ? e.att_vg : e.att_kg) + rc * dkv + kc0 + c, 16u);
  }
  cp_async_commit();
}

// After the copies into `buf` have landed: the anchor (fp32) into key slot
// 15 of the K and V tiles as bf16.
__device__ __forceinline__ void att_anchor_slot(uint8_t* buf, int kvw, int lane) {
  uint8_t* sK = buf;
  uint8_t* sV = buf + kAttKvBytes;
  const float* sA = reinterpret_cast<const float*>(buf + 2 * kAttKvBytes);
  for (int c = lane; c < kvw; c += 32) {
    const uint32_t off = tile_off(kAttAnchor, c >> 3) + (c & 7) * 2;
    *reinterpret_cast<__nv_bfloat16*>(sK + off) = __float2bfloat16_rn(sA[c]);
    *reinterpret_cast<__nv_bfloat16*>(sV + off) = __float2bfloat16_rn(sA[kAttCols + c]);
  }
}

// Starts the copies for the request of the first lane in `lanes` (if any).
__device__ __forceinline__ void att_issue_first(const EpiArgs& e, const AttRow& a, unsigned lanes, int kc0, int kvw,
                                                uint8_t* buf, int lane) {
  if (!lanes) return;
  const int l = __ffs(lanes) - 1;
  const int rc = __shfl_sync(0xffffffffu, a.r, l);
  const int W = __shfl_sync(0xffffffffu, a.W, l);
  const long long base = __shfl_sync(0xffffffffu, a.base, l);
  att_issue(e, rc, W, base, kc0, kvw, buf, lane);
}

// The heads (DH = 64: one, 32: two) of one warp's 32 query rows (q in sQ,
// bf16, 128-byte swizzled rows) against the key slots of each request among
// its rows (rows of other requests get p = 0), one request after another;
// the copies for the next request are started before each request's
// products, those for the next tile's first request (its rows are `nxt`)
// after the last request's products.  Writes the normalised attention output (bf16) into
// the two staging buffers at `stage` (over sQ, once every read of q is done).
template <int DH>
__device__ __forceinline__ void att_tile(const EpiArgs& e, const AttRow& cur, const AttRow& nxt, bool has_next,
                                         int lane, int col0, int kc0, int kvw, int kn0, int kvwn, uint8_t* sQ,
                                         uint8_t* att, int& buf, uint8_t* stage) {
  const int g = lane >> 2, tq = lane & 3;                     // MMA fragment row group / column pair
  const int grp = e.att_group;
  // rows of the fragment slots s = 2 mt + hf (m-tile mt, half hf): 8 s + g
  int rreq[4];
#pragma unroll
  for (int s = 0; s < 4; ++s) rreq[s] = __shfl_sync(0xffffffffu, cur.r, 8 * s + g);
  const uint32_t aQ = smem_u32(sQ);
  const int mi = lane >> 3, rr = lane & 7;                     // ldmatrix: matrix index, row within it
  const float sc = e.att_scale_log2;
  constexpr int hpw = kAttCols / DH;                           // heads of this warp (1 or 2)
  float o[2][8][4];                                            // [m-tile][8-column tile][fragment]
  float lsum[2][2][2];                                         // row sums [head][m-tile][half]
#pragma unroll
  for (int mt = 0; mt < 2; ++mt) {
#pragma unroll
    for (int hl = 0; hl < 2; ++hl) lsum[hl][mt][0] = lsum[hl][mt][1] = 0.f;
#pragma unroll
    for (int n = 0; n < 8; ++n) o[mt][n][0] = o[mt][n][1] = o[mt][n][2] = o[mt][n][3] = 0.f;
  }
  unsigned pending = __ballot_sync(0xffffffffu, cur.r >= 0);
  while (pending) {
    const int leader = __ffs(pending) - 1;
    const int rc = __shfl_sync(0xffffffffu, cur.r, leader);
    const int W = __shfl_sync(0xffffffffu, cur.W, leader);
    pending &= ~__ballot_sync(0xffffffffu, cur.r == rc);
    uint8_t* cb = att + buf * kAttBufBytes;
    cp_async_wait_all();                                      // this request's slots have landed
    __syncwarp();
    att_anchor_slot(cb, kvw, lane);
    // the next copies go to the other buffer, whose last readers (the
    // products of the previous request) are done
    uint8_t* nb = att + (buf ^ 1) * kAttBufBytes;
    if (pending) att_issue_first(e, cur, pending, kc0, kvw, nb, lane);
    __syncwarp();
    const uint32_t aK = smem_u32(cb), aV = aK + kAttKvBytes;
#pragma unroll
    for (int hl = 0; hl < 2; ++hl) {
      if (hl >= hpw) break;
      const int hq = (col0 + hl * DH) / DH;                            // this head (DH: a power of two)
      const int ku = ((grp == 1 ? hq : hq / grp) * DH - kc0) / 8;      // its first K/V unit
      const int qu = hl * DH / 8;                                      // its first query unit
      constexpr int nks = DH / 16;                                     // k-steps of S
      // S = Q K^T: [m-tile][key tile][fragment]
      float sfr[2][2][4];
#pragma unroll
      for (int mt = 0; mt < 2; ++mt)
#pragma unroll
        for (int nt = 0; nt < 2; ++nt) sfr[mt][nt][0] = sfr[mt][nt][1] = sfr[mt][nt][2] = sfr[mt][nt][3] = 0.f;
#pragma unroll
      for (int ks = 0; ks < nks; ++ks) {
        uint32_t kb[4];   // key tile 0 (dims lo, hi), key tile 1 (dims lo, hi)
        ldsm_x4(kb, aK + tile_off((mi >> 1) * 8 + rr, ku + 2 * ks + (mi & 1)));
#pragma unroll
        for (int mt = 0; mt < 2; ++mt) {
          uint32_t qa[4];
          ldsm_x4(qa, aQ + tile_off(16 * mt + (mi & 1) * 8 + rr, qu + 2 * ks + (mi >> 1)));
          mma_16816(sfr[mt][0], qa, kb);
          mma_16816(sfr[mt][1], qa, kb + 2);
        }
      }
      // softmax of each row over its valid slots (window rows below W and
      // the anchor), exp2 of log2-scaled scores; P as the A fragment
      uint32_t pa[2][4];
#pragma unroll
      for (int mt = 0; mt < 2; ++mt) {
#pragma unroll
        for (int hf = 0; hf < 2; ++hf) {
          const bool mine = rreq[2 * mt + hf] == rc;
          float x[4];
#pragma unroll
          for (int i = 0; i < 4; ++i) {
            const int key = (i >> 1) * 8 + 2 * tq + (i & 1);
            x[i] = key < W || key == kAttAnchor ? sfr[mt][i >> 1][2 * hf + (i & 1)] * sc : -INFINITY;
          }
          float mx = fmaxf(fmaxf(x[0], x[1]), fmaxf(x[2], x[3]));
          mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 1));
          mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 2));
          float sum = 0.f;
#pragma unroll
          for (int i = 0; i < 4; ++i) {
            x[i] = mine ? exp2f(x[i] - mx) : 0.f;
            sum += x[i];
          }
          sum += __shfl_xor_sync(0xffffffffu, sum, 1);
          sum += __shfl_xor_sync(0xffffffffu, sum, 2);
          if (mine) lsum[hl][mt][hf] = sum;
          pa[mt][hf] = pack_bf16x2(x[0], x[1]);                  // slots 2 tq, 2 tq + 1
          pa[mt][2 + hf] = pack_bf16x2(x[2], x[3]);              // slots 8 + 2 tq, 9 + 2 tq
        }
      }
      // O += P V over this head's 8-column tiles (two per transposed load)
#pragma unroll
      for (int j = 0; j < DH / 8; j += 2) {
        uint32_t vb[4];   // column tile j (slots 0-7, 8-15), column tile j + 1 (slots 0-7, 8-15)
        ldsm_x4_t(vb, aV + tile_off((mi & 1) * 8 + rr, ku + j + (mi >> 1)));
#pragma unroll
        for (int mt = 0; mt < 2; ++mt) {
          mma_16816(o[mt][qu + j], pa[mt], vb);
          mma_16816(o[mt][qu + j + 1], pa[mt], vb + 2);
        }
      }
    }
    // after the tile's last request: the next tile's first request (its
    // window was looked up during this tile)
    if (!pending && has_next) att_issue_first(e, nxt, __ballot_sync(0xffffffffu, nxt.r >= 0), kn0, kvwn, nb, lane);
    buf ^= 1;
  }
  // no request among this warp's rows (all past M): the next tile's copies
  // (nothing is in flight for this tile)
  if (!__ballot_sync(0xffffffffu, cur.r >= 0) && has_next)
    att_issue_first(e, nxt, __ballot_sync(0xffffffffu, nxt.r >= 0), kn0, kvwn, att + buf * kAttBufBytes, lane);
  // normalise and store: output column 8 n + 2 tq (+1) of rows 16 mt + g and
  // 16 mt + 8 + g into the staging buffers (over q, whose reads are done)
  __syncwarp();
#pragma unroll
  for (int mt = 0; mt < 2; ++mt) {
#pragma unroll
    for (int hf = 0; hf < 2; ++hf) {
      const int orow = 16 * mt + 8 * hf + g;
#pragma unroll
      for (int n = 0; n < 8; ++n) {
        const float l = lsum[(8 * n) / DH][mt][hf];
        const float inv = l > 0.f ? 1.f / l : 0.f;
        const int col = 8 * n + 2 * tq;
        const int cc = col & 31, u = cc >> 3;
        uint8_t* sb = stage + (col >> 5) * 2048;
        *reinterpret_cast<uint32_t*>(sb + orow * 64 + ((u ^ ((orow >> 1) & 3)) << 4) + (cc & 7) * 2) =
            pack_bf16x2(o[mt][n][2 * hf] * inv, o[mt][n][2 * hf + 1] * inv);
      }
    }
  }
}

// The fused epilogue of EPI_ATTN_LG for one epilogue warp over all its tiles
// (TMEM lane quarter q, column half h): per tile, q = acc + b_Q rounded to
// bf16 (the accumulator is released as soon as it has been read), then per
// head the softmax over the request's window rows and anchor of
// q . k / sqrt(d_h) and the weighted values (Sec. 4.1.2 sparse
// cross-attention equation with the local-global key set), stored where q
// would have gone.  The key slots of each tile's first request are copied
// while the previous tile computes; this lane's row request for the next
// tile is read at the start of the current one.  PAIR: tiles of 256 rows on
// a CTA pair, this CTA's 128 rows starting at rank * 128; the accumulator
// is released on rank 0's barrier.
template <bool PAIR>
__device__ __forceinline__ void attn_epilogue_warp(const EpiArgs& e, uint32_t tmem_q, uint64_t* acc_full,
                                                   uint64_t* acc_empty, volatile int* abort_flag, int t_lo, int t_hi,
                                                   int t_step, int n_tiles, int m_tiles, int q, int h,
                                                   const float* bias, const CUtensorMap* tmO, uint8_t* stage,
                                                   uint8_t* att, int rank) {
  constexpr int BNA = 2 * kAttCols;
  constexpr int TM = PAIR ? 2 * BM : BM;
  const int lane = threadIdx.x & 31;
  auto row_of = [&](int t) { return att_tile_m(t, n_tiles, m_tiles, t_step) * TM + rank * BM + q * 32 + lane; };
  auto col_of = [&](int t) { return (t % n_tiles) * BNA + h * kAttCols; };
  // request attended by this lane's row of tile t (-1: past M, or a
  // context-token row, attended by a separate launch)
  auto req_of = [&](int t) {
    return t < t_hi && row_of(t) < e.att_n_cand ? __ldg(e.att_row_req + row_of(t)) : -1;
  };
  // this lane's row in the current tile (cur) and the next (nxt, window
  // looked up during the current tile), and the request of its row two tiles
  // ahead (r2, read during the current tile)
  AttRow cur, nxt;
  int buf = 0;
  if (t_lo < t_hi) {
    cur.r = req_of(t_lo);
    att_row_meta(e, cur);
    int kc0, kvw;
    att_kv_cols(e, col_of(t_lo), kc0, kvw);
    att_issue_first(e, cur, __ballot_sync(0xffffffffu, cur.r >= 0), kc0, kvw, att, lane);
    nxt.r = req_of(t_lo + t_step);
  }
  int i = 0;
  for (int t = t_lo; t < t_hi; t += t_step, ++i) {
    const int b = i & 1;
    const bool has_next = t + t_step < t_hi;
    const int row = row_of(t), col0 = col_of(t);
    const int r2 = req_of(t + 2 * t_step);
    att_row_meta(e, nxt);
    bool go = mbar_wait(acc_full + b, (i >> 1) & 1, abort_flag);
    go = __shfl_sync(0xffffffffu, go ? 1 : 0, 0) != 0;
    if (!go) break;
    tc_fence_after();
    // q = acc + b_Q (bf16) into the staging buffers, free of earlier stores
    if (lane == 0) bulk_wait_read<0>();
    __syncwarp();
    uint8_t* sQ = stage;
    {
      float w[kAttCols];
      tmem_ld64(tmem_q + b * BNA + h * kAttCols, w);
      tc_fence_before();
      __syncwarp();
      if (lane == 0) {                                        // the accumulator may be reused
        if constexpr (PAIR) mbar_arrive_peer_signal(map_peer(acc_empty + b, 0));
        else mbar_arrive(acc_empty + b);
      }
      // every bias read (16-byte aligned columns) before the first store, so
      // the reads are not ordered behind the shared-memory stores
      uint4 pk[kAttCols / 8];
      const float4* b4 = reinterpret_cast<const float4*>(bias + col0);
#pragma unroll
      for (int u = 0; u < kAttCols / 8; ++u) {
        const float4 bl = b4[2 * u], bh = b4[2 * u + 1];
        pk[u].x = pack_bf16x2(w[8 * u] + bl.x, w[8 * u + 1] + bl.y);
        pk[u].y = pack_bf16x2(w[8 * u + 2] + bl.z, w[8 * u + 3] + bl.w);
        pk[u].z = pack_bf16x2(w[8 * u + 4] + bh.x, w[8 * u + 5] + bh.y);
        pk[u].w = pack_bf16x2(w[8 * u + 6] + bh.z, w[8 * u + 7] + bh.w);
      }
#pragma unroll
      for (int u = 0; u < kAttCols / 8; ++u) *reinterpret_cast<uint4*>(sQ + tile_off(lane, u)) = pk[u];
      if (row >= e.att_n_cand && row < e.M) {   // a context-token row: its q for the separate launch
        uint4* qc = reinterpret_cast<uint4*>(static_cast<__nv_bfloat16*>(e.att_q_ctx) +
                                             static_cast<long long>(row) * e.ldo + col0);
#pragma unroll
        for (int u = 0; u < kAttCols / 8; ++u) qc[u] = pk[u];
      }
    }
    __syncwarp();
    int kc0, kvw, kn0 = 0, kvwn = 0;
    att_kv_cols(e, col0, kc0, kvw);
    if (has_next) att_kv_cols(e, col_of(t + t_step), kn0, kvwn);
    if (e.att_dh == 64)
      att_tile<64>(e, cur, nxt, has_next, lane, col0, kc0, kvw, kn0, kvwn, sQ, att, buf, stage);
    else
      att_tile<32>(e, cur, nxt, has_next, lane, col0, kc0, kvw, kn0, kvwn, sQ, att, buf, stage);
    // rows past M hold stale values; the bulk stores of the [M, N] output
    // drop those rows
    fence_async_smem();
    __syncwarp();
    if (lane == 0) {
      tma_store_2d(tmO, stage, col0, row - lane);
      tma_store_2d(tmO, stage + 2048, col0 + 32, row - lane);
      bulk_commit();
    }
    cur = nxt;
    nxt.r = r2;
  }
  cp_async_wait_all();                                        // no copy outlives the kernel's shared memory
  if (lane == 0) bulk_wait_all();
}

// ------------------------------------------------------------------ fused serving attention

// Serving-stream attention of one head for the 32 rows of one warp
// (EPI_SERVE; App. B mask): a candidate row attends to the S context rows of
// its request and to itself.  The tile's accumulator holds q | k | v of the
// head (DH columns each; bias in `bias` at the tile's columns n0 ..); this
// warp takes dims [32 h2, 32 h2 + 32) of each.  The two warps of a lane
// quarter add their partial scores through `red` (slots per row: S context
// keys and the row's own key; `par` alternates the buffer by tile), then
// each forms its 32 output dims: the softmax-weighted context values (bf16,
// from srv_ctx) and the row's own value.
template <int DH>
__device__ __forceinline__ void serve_tile(const EpiArgs& e, uint32_t tacc, int m0, int n0, int head, int h2, int q,
                                           int lane, int par, int r, const float* bias, float* red,
                                           const CUtensorMap* tmO, uint8_t* stage, int& kchunk) {
  const int trow = q * 32 + lane;
  const int row = m0 + trow;
  const bool valid = row < e.M;
  const int S = e.srv_S, d = e.srv_d;
  const int col = 32 * h2;
  const long long ld = 3LL * d;
  const __nv_bfloat16* ctx = static_cast<const __nv_bfloat16*>(e.srv_ctx) + static_cast<long long>(r) * S * ld +
                             head * DH + col;   // q of context row 0; k at + d, v at + 2 d
  float qv[32], kv[32];
  tmem_ld32x2(tacc + col, tacc + DH + col, qv, kv);
  float self = 0.f;
#pragma unroll
  for (int i = 0; i < 32; ++i) {
    qv[i] += bias[n0 + col + i];
    kv[i] += bias[n0 + DH + col + i];
    self = fmaf(qv[i], kv[i], self);
  }
  float part[kSrvSlots];
#pragma unroll
  for (int t = 0; t < kSrvMaxS; ++t) {
    part[t] = 0.f;
    if (t < S) {
      float kc[32];
      load_bf16x32(ctx + t * ld + d, kc);
#pragma unroll
      for (int i = 0; i < 32; ++i) part[t] = fmaf(qv[i], kc[i], part[t]);
    }
  }
  part[kSrvMaxS] = self;
  float* mine = red + ((par * 2 + h2) * 128 + trow) * kSrvSlots;
  const float* other = red + ((par * 2 + (1 - h2)) * 128 + trow) * kSrvSlots;
#pragma unroll
  for (int t = 0; t < kSrvSlots; ++t) mine[t] = part[t];
  named_bar(1 + q, 64);
  float mx = -INFINITY;
#pragma unroll
  for (int t = 0; t < kSrvSlots; ++t) {
    part[t] = (part[t] + other[t]) * e.srv_scale_log2;   // log2-domain scores
    if (t < S || t == kSrvMaxS) mx = fmaxf(mx, part[t]);
  }
  float sum = 0.f;
#pragma unroll
  for (int t = 0; t < kSrvSlots; ++t) {
    part[t] = (t < S || t == kSrvMaxS) ? ex2_approx(part[t] - mx) : 0.f;
    sum += part[t];
  }
  const float inv = 1.f / sum;
  float o[32];
  tmem_ld32(tacc + 2 * DH + col, o);
#pragma unroll
  for (int i = 0; i < 32; ++i) o[i] = (o[i] + bias[n0 + 2 * DH + col + i]) * part[kSrvMaxS];
#pragma unroll
  for (int t = 0; t < kSrvMaxS; ++t) {
    if (t < S) {
      float vc[32];
      load_bf16x32(ctx + t * ld + 2 * d, vc);
#pragma unroll
      for (int i = 0; i < 32; ++i) o[i] = fmaf(part[t], vc[i], o[i]);
    }
  }
#pragma unroll
  for (int i = 0; i < 32; ++i) o[i] *= inv;
  __nv_bfloat16* out =
      valid ? static_cast<__nv_bfloat16*>(e.out) + static_cast<long long>(row) * e.ldo + head * DH + col : nullptr;
  store_chunk<1>(o, out, valid, true, tmO, head * DH + col, m0 + q * 32, stage, kchunk++, lane);
}

// Request of this lane's row of the tile at rows m0.. (0 past M).
__device__ __forceinline__ int serve_req(const EpiArgs& e, int m0, int q, int lane) {
  const int row = m0 + q * 32 + lane;
  return row < e.M ? __ldg(e.srv_row_req + row) : 0;
}

// L1 prefetch of the context keys and values of request r that serve_tile
// reads (head `head`, dims [32 h2, 32 h2 + 32)).
template <int DH>
__device__ __forceinline__ void serve_prefetch(const EpiArgs& e, int r, int head, int h2) {
  const int S = e.srv_S, d = e.srv_d;
  const long long ld = 3LL * d;
  const __nv_bfloat16* ctx =
      static_cast<const __nv_bfloat16*>(e.srv_ctx) + static_cast<long long>(r) * S * ld + head * DH + 32 * h2;
  for (int t = 0; t < S; ++t) {
    prefetch_l1(ctx + t * ld + d);
    prefetch_l1(ctx + t * ld + 2 * d);
  }
}

// ------------------------------------------------------------------ kernel

// BRES: the CTA's whole B slice (BN x K, K <= KRES) stays resident in shared
// memory and only A streams through the ring.  NAP: head actions padded
// (EPI_LN_HEAD).  PAIR: a cluster of two CTAs computes a 256 x BN tile with
// M = 256 MMAs (cta_group::2): each CTA stages its 128 rows of A and half of
// the BN rows of B, so a stage carries half the weight bytes per MMA flop of
// a one-CTA tile.
template <int BN, int EPI, int NAP = 4, bool BRES = false, bool PAIR = false>
struct Shape {
  static constexpr int BN_MMA = BN < 256 ? BN : 256;     // N of one tcgen05.mma
  static constexpr bool SERVE = EPI == EPI_SERVE;
  static constexpr int B_ROWS = PAIR ? BN / 2 : BN;       // rows of B this CTA stages
  static constexpr int B_BOX = PAIR ? B_ROWS : BN_MMA;    // rows of one TMA box of B
  static constexpr int TM = PAIR ? 2 * BM : BM;           // rows of a tile
  static constexpr int KRES = 256;
  static constexpr int BRES_BYTES = BRES ? BN * KRES * 2 : 0;
  static constexpr int B_STAGE_BYTES = BRES ? 0 : B_ROWS * BK * 2;
  static constexpr int STAGE_BYTES = A_STAGE_BYTES + B_STAGE_BYTES;
  static constexpr bool LN = EPI == EPI_LN || EPI == EPI_LN_HEAD;
  static constexpr int RED_BYTES = LN ? 2 * 128 * kRedStride * 4 : SERVE ? 2 * 2 * 128 * kSrvSlots * 4 : 0;
  static constexpr int WEFF_BYTES = EPI == EPI_LN_HEAD ? BN * NAP * 4 : 0;
  // bias [kStageN] floats ([kStageNRes] with BRES), then (cache-row remap) offsets and
  // first rows; rounded to 1 KB so that the staging buffers after it start on
  // a swizzle-atom boundary
  static constexpr bool ATT = EPI == EPI_ATTN_LG;
  // 256-column tiles streaming both operands (the K/V build, the QKV and FFN
  // projections at d = 512): one bulk-store staging buffer per warp and the
  // bias read through L1 leave room for a fourth operand stage
  static constexpr bool LEAN = !BRES && !LN && !ATT && BN == 256;
  static constexpr int SBUF = (LEAN || SERVE) ? 1 : 2;    // bulk-store staging buffers per warp
  // (the fused attention on pairs reads its bias through L1: the room is a
  // fifth operand stage)
  static constexpr int STAGE_N = BRES ? kStageNRes : SERVE ? kStageNSrv : (ATT && PAIR) ? 0
                                 : (ATT || LEAN) ? kStageNAtt : kStageN;
  static constexpr int AUX_BYTES =
      LN ? 0 : (((STAGE_N * 4) + (EPI == EPI_KV ? (2 * kStageSeg + 1) * 4 : 0) + 1023) / 1024) * 1024;
  // fused attention: each epilogue warp's staged window and anchor (fp32)
  static constexpr int ATT_BYTES = ATT ? kEpiWarps * kAttWarpBytes : 0;
  // bulk-store staging: two 2 KB buffers per epilogue warp (bf16 outputs)
  static constexpr int STG_BYTES = EPI == EPI_LN_HEAD ? 0 : kEpiWarps * SBUF * 2048;
  static constexpr int EXTRA = BRES_BYTES + RED_BYTES + WEFF_BYTES + AUX_BYTES + STG_BYTES + ATT_BYTES + 1024 + 256;
  static constexpr int STAGES_FIT = (227 * 1024 - EXTRA) / STAGE_BYTES;
  static constexpr int STAGES = STAGES_FIT > 8 ? 8 : STAGES_FIT;
  static constexpr int ACC_BUFS = BN <= 256 ? 2 : 1;      // TMEM double buffer
  static constexpr int TMEM_USED = BN * ACC_BUFS;
  static constexpr int TMEM_COLS = TMEM_USED <= 32 ? 32 : TMEM_USED <= 64 ? 64 : TMEM_USED <= 128 ? 128
                                   : TMEM_USED <= 256 ? 256 : 512;   // a power of two
  static constexpr int SMEM_BYTES = STAGES * STAGE_BYTES + EXTRA;
  static_assert(STAGES >= 2, "pipeline depth");
  static_assert(!(BRES && LN), "resident B only for the plain epilogues");
  static_assert((RED_BYTES + WEFF_BYTES + AUX_BYTES) % 1024 == 0 || STG_BYTES == 0,
                "staging buffers need 512-byte alignment (64-byte swizzle atoms)");
  static_assert((RED_BYTES + WEFF_BYTES + AUX_BYTES + STG_BYTES + ATT_BYTES) % 16 == 0,
                "mbarriers must stay 8-byte aligned");
  static_assert(!ATT || (BN == 2 * kAttCols && !BRES), "fused attention: 128-column tiles");
  static_assert(!PAIR || (LEAN && BN == 256) || (SERVE && BN == 192) || (ATT && BN == 128),
                "CTA pairs: 256-column streaming tiles and the fused attentions");
  static_assert(!SERVE || PAIR, "fused serving attention: CTA pairs");
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

template <int BN, int EPI, int NAP, bool BRES, bool PAIR>
__global__ void __launch_bounds__(NUM_THREADS, 1)
    gemm_tc_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                   const __grid_constant__ CUtensorMap tmO, const EpiArgs e,
                   const __grid_constant__ ParamsFor<EPI> kp) {
  using S = Shape<BN, EPI, NAP, BRES, PAIR>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* sA = smem;
  uint8_t* sB = smem + S::STAGES * A_STAGE_BYTES;
  uint8_t* sBres = sB + S::STAGES * S::B_STAGE_BYTES;
  float* red = reinterpret_cast<float*>(sBres + S::BRES_BYTES);
  float* s_weff = reinterpret_cast<float*>(reinterpret_cast<uint8_t*>(red) + S::RED_BYTES);
  float* s_bias = reinterpret_cast<float*>(reinterpret_cast<uint8_t*>(s_weff) + S::WEFF_BYTES);
  int* s_seg = reinterpret_cast<int*>(s_bias + S::STAGE_N);
  int* s_dst = s_seg + kStageSeg + 1;
  uint8_t* s_stage = reinterpret_cast<uint8_t*>(s_bias) + S::AUX_BYTES;
  uint8_t* s_att = s_stage + S::STG_BYTES;
  uint64_t* full = reinterpret_cast<uint64_t*>(s_att + S::ATT_BYTES);
  uint64_t* empty = full + S::STAGES;
  uint64_t* acc_full = empty + S::STAGES;
  uint64_t* acc_empty = acc_full + 2;
  uint64_t* b_full = acc_empty + 2;     // resident B slice loaded
  uint64_t* b_empty = b_full + 1;       // last MMA reading the resident B slice done
  uint32_t* tmem_holder = reinterpret_cast<uint32_t*>(b_empty + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_holder + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  // PAIR: rank 1 holds rows [128, 256) of every tile; rank 0 issues the MMAs
  // and owns the barriers that gate them (full, acc_empty)
  const uint32_t rank = PAIR ? cluster_rank() : 0;
  const int n_tiles = e.N / BN;
  const int m_tiles = (e.M + S::TM - 1) / S::TM;
  const int num_tiles = m_tiles * n_tiles;
  const int num_kb = e.K / BK;
  // this CTA's tiles: t_lo, t_lo + t_step, ... < t_hi (the same for both CTAs of a pair)
  int t_lo = PAIR ? blockIdx.x / 2 : blockIdx.x, t_hi = num_tiles, t_step = PAIR ? gridDim.x / 2 : gridDim.x;
  if constexpr (BRES) {
    t_lo = static_cast<int>(static_cast<long long>(blockIdx.x) * num_tiles / gridDim.x);
    t_hi = static_cast<int>(static_cast<long long>(blockIdx.x + 1) * num_tiles / gridDim.x);
    t_step = 1;
  }
  auto tile_n = [&](int t) { return BRES ? t / m_tiles : t % n_tiles; };
  auto tile_m = [&](int t) {
    return BRES ? t % m_tiles : S::ATT ? att_tile_m(t, n_tiles, m_tiles, t_step) : t / n_tiles;
  };

  if (threadIdx.x == 0) {
    for (int s = 0; s < S::STAGES; ++s) {
      mbar_init(full + s, 1);
      mbar_init(empty + s, 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(acc_full + b, 1);
      mbar_init(acc_empty + b, PAIR ? 2 * kEpiWarps : kEpiWarps);   // rank 0's: both CTAs' epilogues
    }
    mbar_init(b_full, 1);
    mbar_init(b_empty, 1);
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 1) {
    if constexpr (PAIR) tmem_alloc_pair(tmem_holder, S::TMEM_COLS);
    else tmem_alloc(tmem_holder, S::TMEM_COLS);
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_holder;
  if constexpr (PAIR) cluster_sync();   // both CTAs' barriers exist before any crosses the pair
  // shared::cluster address of rank 0's copy of a barrier (PAIR)
  auto lead = [&](uint64_t* bar) { return PAIR ? map_peer(bar, 0) : smem_u32(bar); };
  // bytes that complete one stage: both CTAs' loads count on rank 0's barrier
  constexpr uint32_t kFullBytes = (PAIR ? 2 : 1) * S::STAGE_BYTES;
  const bool expects = !PAIR || rank == 0;
  auto load_a = [&](int s, int kb, int m0) {
    if constexpr (PAIR) tma_load_2d_pair(sA + s * A_STAGE_BYTES, &tmA, lead(full + s), kb * BK, m0);
    else tma_load_2d(sA + s * A_STAGE_BYTES, &tmA, full + s, kb * BK, m0);
  };
  auto load_b = [&](int s, int kb, int n0) {
#pragma unroll
    for (int j = 0; j < S::B_ROWS; j += S::B_BOX) {
      if constexpr (PAIR)
        tma_load_2d_pair(sB + s * S::B_STAGE_BYTES + j * (BK * 2), &tmB, lead(full + s), kb * BK,
                         n0 + static_cast<int>(rank) * S::B_ROWS + j);
      else
        tma_load_2d(sB + s * S::B_STAGE_BYTES + j * (BK * 2), &tmB, full + s, kb * BK, n0 + j);
    }
  };
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
        if (expects) mbar_expect_tx(full + kb, kFullBytes);
        load_b(kb, kb, n0);
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
    if (e.N <= S::STAGE_N) {
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
        const int m0 = tile_m(t) * S::TM + static_cast<int>(rank) * BM, n0 = tile_n(t) * BN;
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
            load_a(s, kb, m0);
            continue;
          }
          if (!mbar_wait(empty + s, ph ^ 1, abort_flag)) {
            ok = false;
            break;
          }
          if (expects) mbar_expect_tx(full + s, kFullBytes);
          load_a(s, kb, m0);
          if constexpr (!BRES) load_b(s, kb, n0);
        }
      }
      if constexpr (PAIR) {
        // rank 0's MMAs release this CTA's stages by multicast commits: take
        // the last ones before the CTA may exit
        for (int k = it > S::STAGES ? it - S::STAGES : 0; k < it && !*abort_flag; ++k)
          mbar_wait(empty + k % S::STAGES, (k / S::STAGES) & 1, abort_flag);
      }
      if (*abort_flag && expects) {
        // let the copies already in flight land before shared memory is released
        for (int k = it > S::STAGES ? it - S::STAGES : 0; k < it; ++k)
          mbar_wait_plain(full + k % S::STAGES, (k / S::STAGES) & 1);
        if (BRES && nb > 0) mbar_wait_plain(b_full, (nb - 1) & 1);
      }
    }
  } else if (warp == 1) {
    if (lane == 0 && (!PAIR || rank == 0)) {
      constexpr uint32_t idesc = idesc_bf16(S::TM, S::BN_MMA);
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
              if constexpr (PAIR)
                mma_bf16_pair(dacc + j * S::BN_MMA, adesc + 2 * k, bdesc + boff + 2 * k, idesc,
                              (kb > 0 || k > 0) ? 1u : 0u);
              else
                mma_bf16(dacc + j * S::BN_MMA, adesc + 2 * k, bdesc + boff + 2 * k, idesc,
                         (kb > 0 || k > 0) ? 1u : 0u);
            }
          }
          if constexpr (PAIR) mma_commit_pair(empty + s, 3);
          else mma_commit(empty + s);
        }
        // also on abort: the epilogue waits on every issued MMA
        if constexpr (PAIR) mma_commit_pair(acc_full + buf, 3);
        else mma_commit(acc_full + buf);
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
    uint8_t* stage = s_stage + ew * S::SBUF * 2048;
    if constexpr (S::ATT) {
      attn_epilogue_warp<PAIR>(e, tmem + (static_cast<uint32_t>(q * 32) << 16), acc_full, acc_empty, abort_flag,
                               t_lo, t_hi, t_step, n_tiles, m_tiles, q, h, bias, &tmO, stage,
                               s_att + ew * kAttWarpBytes, static_cast<int>(rank));
    } else if constexpr (S::SERVE) {
      int kchunk = 0;
      int i = 0;
      // Each tile's row requests are read two tiles ahead and its context
      // rows prefetched into L1 one tile ahead, so no tile waits on a chain
      // of dependent global loads.
      auto rows_of = [&](int t) { return tile_m(t) * S::TM + static_cast<int>(rank) * BM; };
      int r_cur = t_lo < t_hi ? serve_req(e, rows_of(t_lo), q, lane) : 0;
      int r_next = t_lo + t_step < t_hi ? serve_req(e, rows_of(t_lo + t_step), q, lane) : 0;
      if (t_lo < t_hi) serve_prefetch<BN / 3>(e, r_cur, tile_n(t_lo), h);
      for (int t = t_lo; t < t_hi; t += t_step, ++i) {
        const int buf = i % S::ACC_BUFS;
        const uint32_t use = i / S::ACC_BUFS;
        const int r = r_cur;
        r_cur = r_next;
        r_next = t + 2 * t_step < t_hi ? serve_req(e, rows_of(t + 2 * t_step), q, lane) : 0;
        if (t + t_step < t_hi) serve_prefetch<BN / 3>(e, r_cur, tile_n(t + t_step), h);
        bool go = mbar_wait(acc_full + buf, use & 1, abort_flag);
        go = __shfl_sync(0xffffffffu, go ? 1 : 0, 0) != 0;
        if (!go) break;
        tc_fence_after();
        const int m0 = rows_of(t), hd = tile_n(t);
        serve_tile<BN / 3>(e, tmem + buf * BN + (static_cast<uint32_t>(q * 32) << 16), m0, hd * BN, hd, h, q, lane,
                           i & 1, r, bias, red, &tmO, stage, kchunk);
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive_peer_signal(lead(acc_empty + buf));
      }
      if (lane == 0) bulk_wait_all();
    } else {
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
        const int m0 = tile_m(t) * S::TM + static_cast<int>(rank) * BM, n0 = tile_n(t) * BN;
        epilogue<BN, EPI, NAP, S::SBUF>(e, tmem + buf * BN + (static_cast<uint32_t>(q * 32) << 16), m0 + q * 32 + lane, n0,
                               h * (BN / 2), q, h, red, s_weff, bias, seg_off, dst_row0, &tmO, stage, kchunk);
        tc_fence_before();
        __syncwarp();
        if (lane == 0) {
          if constexpr (PAIR) mbar_arrive_peer_signal(lead(acc_empty + buf));
          else mbar_arrive(acc_empty + buf);
        }
      }
      if (lane == 0) bulk_wait_all();   // this warp's bulk stores are complete before exit
    }
  }
  tc_fence_before();
  __syncthreads();
  // PAIR: rank 1's epilogue arrivals on rank 0 have landed and neither CTA
  // frees its TMEM before the other is done with the pair's accumulators
  if constexpr (PAIR) cluster_sync();
  if (warp == 1) {
    tc_fence_after();
    if constexpr (PAIR) tmem_dealloc_pair(tmem, S::TMEM_COLS);
    else tmem_dealloc(tmem, S::TMEM_COLS);
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

template <int BN, int EPI, int NAP = 4, bool BRES = false, bool PAIR = false>
static cudaError_t launch_bn(const __nv_bfloat16* A, long long lda, const __nv_bfloat16* B, const EpiArgs& e,
                             cudaStream_t s, int cls) {
  using Sh = Shape<BN, EPI, NAP, BRES, PAIR>;
  auto kern = gemm_tc_kernel<BN, EPI, NAP, BRES, PAIR>;
  if (BRES && e.K > Sh::KRES) return cudaErrorInvalidValue;
  static int max_ctas = 0;   // CTAs resident at once (whole pairs with PAIR)
  if (!max_ctas) {
    cudaError_t err = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, Sh::SMEM_BYTES);
    if (err != cudaSuccess) return err;
    int n = num_sms();
    if (PAIR) {
      cudaLaunchAttribute at[1];
      at[0].id = cudaLaunchAttributeClusterDimension;
      at[0].val.clusterDim.x = 2;
      at[0].val.clusterDim.y = 1;
      at[0].val.clusterDim.z = 1;
      cudaLaunchConfig_t q = {};
      q.gridDim = dim3((num_sms() / 2) * 2);
      q.blockDim = dim3(NUM_THREADS);
      q.dynamicSmemBytes = Sh::SMEM_BYTES;
      q.attrs = at;
      q.numAttrs = 1;
      int c = 0;
      if (cudaOccupancyMaxActiveClusters(&c, kern, &q) != cudaSuccess || c <= 0) {
        (void)cudaGetLastError();
        c = num_sms() / 2;
      }
      n = 2 * c;
    }
    max_ctas = n;
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
  } else if (EPI == EPI_SERVE) {
    if (!make_tmap_out(&to, e.out, e.M, e.N / 3, e.ldo)) return cudaErrorInvalidValue;   // one head's d_h per tile
  } else {
    if (!make_tmap_out(&to, e.out, e.M, e.N, e.ldo)) return cudaErrorInvalidValue;
  }
  const long long tiles = static_cast<long long>((e.M + Sh::TM - 1) / Sh::TM) * (e.N / BN);
  const int per_tile = PAIR ? 2 : 1;
  const int grid = static_cast<int>(tiles * per_tile < max_ctas ? tiles * per_tile : (max_ctas / per_tile) * per_tile);
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
  cudaError_t err;
  if constexpr (PAIR) {
    cudaLaunchAttribute at[2];
    at[0].id = cudaLaunchAttributeClusterDimension;
    at[0].val.clusterDim.x = 2;
    at[0].val.clusterDim.y = 1;
    at[0].val.clusterDim.z = 1;
    at[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    at[1].val.programmaticStreamSerializationAllowed = 1;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(grid);
    cfg.blockDim = dim3(NUM_THREADS);
    cfg.dynamicSmemBytes = Sh::SMEM_BYTES;
    cfg.stream = s;
    cfg.attrs = at;
    cfg.numAttrs = 2;
    err = cudaLaunchKernelEx(&cfg, kern, ta, tb, to, e, kp);
  } else {
    err = launch_pdl(kern, dim3(grid), dim3(NUM_THREADS), Sh::SMEM_BYTES, s, ta, tb, to, e, kp);
  }
  prof_end(cls, s);
  return err;
}

bool tc_gemm_supported(int N, int K, int epi) {
  if (K <= 0 || K % BK != 0 || N <= 0) return false;
  if (epi == EPI_LN || epi == EPI_LN_HEAD) return N == 64 || N == 128 || N == 256 || N == 512;
  if (epi == EPI_ATTN_LG) return N % 128 == 0 && N <= kStageNAtt;
  if (epi == EPI_SERVE) return N % 192 == 0 && N <= kStageNSrv;
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
  // long streams of 256-column tiles: CTA pairs with M = 256 MMAs
  if (fits(256) && ((e.M + 255) / 256) * (e.N / 256) >= num_sms())
    return launch_bn<256, EPI, 4, false, true>(A, lda, B, e, s, cls);
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
    case EPI_ATTN_LG:
      if ((e.att_dh != 32 && e.att_dh != 64) || e.att_l_local < 0 || e.att_l_local > kAttWinMax ||
          e.att_group < 1 || e.att_dkv % 8 != 0)
        return cudaErrorNotSupported;
      // long streams of row tiles: CTA pairs (M = 256 MMAs, half the weight
      // bytes per CTA, five operand stages)
      if (((e.M + 255) / 256) * (e.N / 128) >= num_sms())
        return launch_bn<128, EPI_ATTN_LG, 4, false, true>(A, lda, B, e, s, cls);
      return launch_bn<128, EPI_ATTN_LG>(A, lda, B, e, s, cls);
    case EPI_SERVE:
      if (e.srv_S < 0 || e.srv_S > kSrvMaxS || e.N != 3 * e.srv_d) return cudaErrorNotSupported;
      return launch_bn<192, EPI_SERVE, 4, false, true>(A, lda, B, e, s, cls);
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
