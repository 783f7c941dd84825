// Projections of the DiT block: C[M,N] = A[M,K] W[N,K]^T with a fused epilogue.
//
// bf16 operands run on the 5th-generation tensor cores: a persistent, warp-specialised
// kernel with one TMA producer warp, one MMA-issuing warp and four epilogue warps.
// Operand tiles (128 x 64 of A, BN x 64 of W, 128-byte swizzle) stream through a
// multi-stage shared-memory ring guarded by mbarriers; tcgen05.mma accumulates a
// 128 x BN fp32 tile in tensor memory, double-buffered so the epilogue of one tile
// overlaps the main loop of the next.  fp32 operands (the fp32 configuration, which
// must hold 1e-4 relative parity) use a CUDA-core kernel with the same epilogue.
#include <algorithm>
#include <cstdio>
#include <mutex>

#include "common.cuh"
#include "epilogue.cuh"
#include "kernels.h"

namespace bag {

// ---------------------------------------------------------------------------
// TMA descriptor encoding through the driver entry point
// ---------------------------------------------------------------------------
typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                  const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                  const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

static EncodeTiledFn get_encode_fn() {
  static EncodeTiledFn fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(p);
  });
  return fn;
}

int encode_tmap_2d_bf16(CUtensorMap* map, const void* base, uint64_t inner, uint64_t outer,
                        uint64_t row_stride_bytes, uint32_t box_inner, uint32_t box_outer) {
  EncodeTiledFn fn = get_encode_fn();
  if (!fn) return -1;
  cuuint64_t dims[2] = {inner, outer};
  cuuint64_t strides[1] = {row_stride_bytes};
  cuuint32_t box[2] = {box_inner, box_outer};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims,
                  strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                  CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS ? 0 : (int)r;
}

static int num_sms() {
  static int n = 0;
  if (n == 0) {
    int dev = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
    if (n <= 0) n = 148;
  }
  return n;
}

// ---------------------------------------------------------------------------
// CUDA-core GEMM (fp32 or bf16 operands, fp32 accumulation)
// ---------------------------------------------------------------------------
template <typename T>
BAG_DEV float ld_f(const T* p) {
  if constexpr (sizeof(T) == 2)
    return __bfloat162float(*reinterpret_cast<const __nv_bfloat16*>(p));
  else
    return *p;
}

template <typename T>
__global__ void __launch_bounds__(256) gemm_simt_kernel(const T* __restrict__ A, long lda,
                                                        const T* __restrict__ W, long ldw,
                                                        int M, int N, int K, const Epi e) {
  grid_dep_sync();
  if (epi_skip(e.st, e.flag_want)) return;
  const int t = epi_step(e);
  __shared__ float As[16][64 + 4];
  __shared__ float Ws[16][64 + 4];
  const int tx = threadIdx.x % 16, ty = threadIdx.x / 16;
  const int m0 = blockIdx.y * 64, n0 = blockIdx.x * 64;
  float acc[4][4];
#pragma unroll
  for (int i = 0; i < 4; ++i)
#pragma unroll
    for (int j = 0; j < 4; ++j) acc[i][j] = 0.f;
  for (int k0 = 0; k0 < K; k0 += 16) {
    for (int i = threadIdx.x; i < 1024; i += 256) {
      const int r = i / 16, c = i % 16;
      const int m = m0 + r, n = n0 + r, k = k0 + c;
      As[c][r] = (m < M && k < K) ? ld_f(A + (long)m * lda + k) : 0.f;
      Ws[c][r] = (n < N && k < K) ? ld_f(W + (long)n * ldw + k) : 0.f;
    }
    __syncthreads();
#pragma unroll
    for (int kk = 0; kk < 16; ++kk) {
      float a[4], b[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) a[i] = As[kk][ty * 4 + i];
#pragma unroll
      for (int j = 0; j < 4; ++j) b[j] = Ws[kk][tx * 4 + j];
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) acc[i][j] += a[i] * b[j];
    }
    __syncthreads();
  }
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int row = m0 + ty * 4 + i;
    const int col = n0 + tx * 4;
    if (row < M && col < N) epi_apply<4>(e, t, row, col, acc[i]);
  }
}

// ---------------------------------------------------------------------------
// tcgen05 GEMM
// ---------------------------------------------------------------------------
constexpr int TC_BM = 128, TC_BK = 64;

// Tile order within one problem: groups of G row tiles, each group visiting every
// column tile with the row tile varying fastest.  A wave of tiles then shares at most G
// row tiles of A (which stay in L2 while the group walks the columns) instead of
// streaming all of A once per column tile; G comes from the L2 share one group's rows
// may take (tile_group_rows).
BAG_DEV void raster(int l, int num_m, int num_n, int G, int& mt, int& nt) {
  const int per_group = G * num_n;
  const int g = l / per_group;
  const int idx = l - g * per_group;
  const int gm = min(G, num_m - g * G);
  mt = g * G + idx % gm;
  nt = idx / gm;
}

#ifndef BAG_TILE_GROUP_L2_MB
#define BAG_TILE_GROUP_L2_MB 40
#endif
// Row tiles per group: as many BM-row slices of A (K bf16 columns, twice as many for a
// split A) as fit in the L2 share, at least 1, at most all of them.
static int tile_group_rows(int M, int BM, int K, int a_split) {
  const int num_m = (M + BM - 1) / BM;
  if (num_m <= 0) return 1;
  const double slice = (double)BM * K * 2.0 * (a_split ? 2 : 1);
  const int g = (int)((double)BAG_TILE_GROUP_L2_MB * 1048576.0 / slice);
  return std::max(1, std::min(num_m, g));
}

// Per epilogue warp: a 32 x 33-word shared-memory tile for transposing V.
constexpr int kVtScratchFloats = 32 * 33;
constexpr int kVtScratchBytes = 4 * kVtScratchFloats * 4;  // four epilogue warps

BAG_DEV uint16_t to16(float x, bool f16) {
  return f16 ? __half_as_ushort(__float2half_rn(x)) : __bfloat16_as_ushort(__float2bfloat16_rn(x));
}
BAG_DEV uint32_t pack16x2(float a, float b, bool f16) { return f16 ? pack_f16x2(a, b) : pack_bf16x2(a, b); }

// 32 consecutive 16-bit tokens of one V^T row starting at dst: 16-byte stores when dst is
// 16-byte aligned, else 4-byte stores (with a single leading element when dst is odd).
BAG_DEV void store_vt_run(uint16_t* dst, const float* tc, bool f16) {
  if ((reinterpret_cast<uintptr_t>(dst) & 15) == 0) {
#pragma unroll
    for (int k = 0; k < 32; k += 8) {
      uint4 w;
      w.x = pack16x2(tc[k], tc[k + 1], f16);
      w.y = pack16x2(tc[k + 2], tc[k + 3], f16);
      w.z = pack16x2(tc[k + 4], tc[k + 5], f16);
      w.w = pack16x2(tc[k + 6], tc[k + 7], f16);
      *reinterpret_cast<uint4*>(dst + k) = w;
    }
  } else if ((reinterpret_cast<uintptr_t>(dst) & 3) == 0) {
#pragma unroll
    for (int k = 0; k < 32; k += 2) *reinterpret_cast<uint32_t*>(dst + k) = pack16x2(tc[k], tc[k + 1], f16);
  } else {
    dst[0] = to16(tc[0], f16);
#pragma unroll
    for (int k = 1; k < 31; k += 2) *reinterpret_cast<uint32_t*>(dst + k) = pack16x2(tc[k], tc[k + 1], f16);
    dst[31] = to16(tc[31], f16);
  }
}

// V columns of a QKV projection with 16-bit (bf16 or fp16) storage, stored transposed per head
// (vt[(head * dh + e) * vpad + token]): the warp's 32 rows x 32 columns pass through
// shared memory, so each lane writes one column's 32 consecutive tokens as four 16-byte
// stores instead of 32 two-byte stores.  Rows past M (the last tile) and token offsets
// that are not 16-byte aligned take per-element stores.
BAG_DEV void store_vt_warp(const Epi& e, int row, int col, float* v, float* sbuf) {
  const int lane = threadIdx.x & 31;
  if (e.bias) {
#pragma unroll
    for (int j = 0; j < 32; ++j) v[j] += __ldg(e.bias + col + j);
  }
#pragma unroll
  for (int j = 0; j < 32; ++j) sbuf[j * 33 + lane] = v[j];
  __syncwarp();
  float tc[32];
#pragma unroll
  for (int k = 0; k < 32; ++k) tc[k] = sbuf[lane * 33 + k];
  __syncwarp();
  const int row0 = row - lane;
  // guidance branches (br_rows > 0): the warp's 32 rows take the fast path only when
  // they all belong to one branch
  const bool br1 = e.br_rows > 0 && row0 >= e.br_rows;
  const bool one_branch = e.br_rows == 0 || br1 || row0 + 31 < e.br_rows;
  const int jr0 = row0 - (br1 ? e.br_rows : 0) + e.row_off;
  const int cc = col + e.col_base - 2 * e.d + lane;  // this lane's column within V
  const bool f16 = e.qkv_type == kStoreF16;
  uint16_t* vbase = reinterpret_cast<uint16_t*>(e.v);
  uint16_t* dst = vbase + (br1 ? e.br_vt : 0) + (long)cc * e.vpad + jr0;
  if (row0 + 31 < e.M && one_branch) {
    store_vt_run(dst, tc, f16);
  } else {
#pragma unroll
    for (int k = 0; k < 32; ++k) {
      const int rk = row0 + k;
      if (rk < e.M) {
        const bool b1 = e.br_rows > 0 && rk >= e.br_rows;
        const long at = (b1 ? e.br_vt : 0) + (long)cc * e.vpad + rk - (b1 ? e.br_rows : 0) + e.row_off;
        vbase[at] = to16(tc[k], f16);
      }
    }
  }
}

// One thread's row of a BN-column accumulator in TMEM (lane base already in tb) through
// the epilogue, columns col0 .. col0 + BN - 1.  vt_buf: this warp's transpose tile.
template <int BN>
BAG_DEV void drain_accumulator(const Epi& e, int t, int row, int col0, uint32_t tb, float* vt_buf) {
  const bool vt_warp = e.kind == EPI_QKV && e.v_mode == 1 && e.qkv_type != kStoreF32;
  if (e.qn_q) {
    // QK-norm: the tile holds whole heads (BN a multiple of dh, checked at launch); a
    // first pass over each q / k head takes its sum of squares (bias included), the
    // second applies the epilogue with 1 / RMS.  The TMEM loads are warp-wide, so every
    // lane takes them whatever its row.
    const int dh = e.dh;
#pragma unroll 1
    for (int h0 = 0; h0 < BN; h0 += dh) {
      const int col = col0 + h0;
      float rs = 1.f;
      if ((col + e.col_base) / e.d < 2 && col < e.N) {
        float ss = 0.f;
#pragma unroll 1
        for (int c = 0; c < dh; c += 32) {
          float v[32];
          tmem_ld32(tb + (uint32_t)(h0 + c), v);
#pragma unroll
          for (int j = 0; j < 32; ++j) {
            const float x = v[j] + (e.bias ? __ldg(e.bias + col + c + j) : 0.f);
            ss = fmaf(x, x, ss);
          }
        }
        rs = rsqrtf(ss / (float)dh + 1e-6f);
      }
#pragma unroll 1
      for (int c = 0; c < dh; c += 32) {
        float v[32];
        tmem_ld32(tb + (uint32_t)(h0 + c), v);
        if (vt_warp && col + c < e.N && (col + c + e.col_base) / e.d == 2)
          store_vt_warp(e, row, col + c, v, vt_buf);
        else
          epi_apply<32>(e, t, row, col + c, v, rs);
      }
    }
  } else {
#pragma unroll 1
    for (int c = 0; c < BN / 32; ++c) {
      float v[32];
      tmem_ld32(tb + (uint32_t)(c * 32), v);
      const int col = col0 + c * 32;
      if (vt_warp && col < e.N && (col + e.col_base) / e.d == 2)
        store_vt_warp(e, row, col, v, vt_buf);  // warp-uniform branch
      else
        epi_apply<32>(e, t, row, col, v);
    }
  }
}

template <int BN>
struct TcCfg {
  static constexpr int STAGES = BN == 256 ? 4 : (BN == 128 ? 6 : 8);
  static constexpr int A_BYTES = TC_BM * TC_BK * 2;
  static constexpr int B_BYTES = BN * TC_BK * 2;
  static constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
  static constexpr int TMEM_COLS = 2 * BN;
  static constexpr int SMEM = STAGES * STAGE_BYTES + 1024 + 256 + kVtScratchBytes;
};

template <int BN>
__global__ void __launch_bounds__(192, 1)
    gemm_tc_kernel(const __grid_constant__ CUtensorMap tmA0, const __grid_constant__ CUtensorMap tmB0,
                   const __grid_constant__ CUtensorMap tmA1, const __grid_constant__ CUtensorMap tmB1,
                   const __grid_constant__ Epi e0, const __grid_constant__ Epi e1, int M0, int M1,
                   int N, int K, int a_split, int g0, int g1, int* err) {
  grid_dep_sync();
  // Two independent problems with the same N and K may share one launch (problem 1 has
  // M1 rows, possibly 0): their tiles form one list, problem 0's first, so a small
  // problem fills the SMs the large one leaves idle in its last wave.
  using C = TcCfg<BN>;
  if (epi_skip(e0.st, e0.flag_want)) return;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  uint8_t* sA = smem;
  uint8_t* sB = smem + C::STAGES * C::A_BYTES;
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + C::STAGES * C::STAGE_BYTES);
  uint64_t* empty = full + C::STAGES;
  uint64_t* tfull = empty + C::STAGES;
  uint64_t* tempty = tfull + 2;
  uint64_t* drain = tempty + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain + 1);
  float* vt_scratch = reinterpret_cast<float*>(smem + C::STAGES * C::STAGE_BYTES + 256);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
  const int num_m0 = (M0 + TC_BM - 1) / TC_BM, num_m1 = (M1 + TC_BM - 1) / TC_BM, num_n = N / BN;
  const int tiles0 = num_m0 * num_n;
  auto decode = [&](int tile, int& pb, int& mt, int& nt) {
    if (tile < tiles0) {
      pb = 0;
      raster(tile, num_m0, num_n, g0, mt, nt);
    } else {
      pb = 1;
      raster(tile - tiles0, num_m1, num_n, g1, mt, nt);
    }
  };
  // a_split: A holds [hi | lo] bf16 halves of an fp32 activation ([M, 2K]); the K loop
  // runs twice as long, feeding each W chunk once with hi and once with lo, so the
  // product is accurate to fp32 accumulation while W is streamed once.
  const int tiles = tiles0 + num_m1 * num_n, kit = (a_split ? 2 : 1) * (K / TC_BK);
  const int t = epi_step(e0);

  if (threadIdx.x == 0) {
    for (int s = 0; s < C::STAGES; ++s) {
      mbar_init(full + s, 1);
      mbar_init(empty + s, 1);
    }
    mbar_init(tfull, 1);
    mbar_init(tfull + 1, 1);
    mbar_init(tempty, 128);
    mbar_init(tempty + 1, 128);
    mbar_init(drain, 1);
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == 0 && lane == 0) {
    tma_prefetch_desc(&tmA0);
    tma_prefetch_desc(&tmB0);
    if (M1 > 0) {
      tma_prefetch_desc(&tmA1);
      tma_prefetch_desc(&tmB1);
    }
  }
  if (warp == 1) {
    tmem_alloc(tmem_slot, C::TMEM_COLS);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;

  if (warp == 0) {
    if (lane == 0) {
      // ---------------- TMA producer ----------------
      int s = 0;
      uint32_t ph = 0;
      long issued = 0;
      bool ok = true;
      for (int tile = blockIdx.x; tile < tiles && ok; tile += gridDim.x) {
        int pb, mt, nt;
        decode(tile, pb, mt, nt);
        const CUtensorMap* tmA = pb ? &tmA1 : &tmA0;
        const CUtensorMap* tmB = pb ? &tmB1 : &tmB0;
        for (int kb = 0; kb < kit; ++kb) {
          if (!mbar_wait(empty + s, ph ^ 1, abort_flag)) {
            ok = false;
            break;
          }
          mbar_arrive_expect_tx(full + s, C::STAGE_BYTES);
          const int ka = a_split ? (kb & 1) * K + (kb >> 1) * TC_BK : kb * TC_BK;
          const int kw = a_split ? (kb >> 1) * TC_BK : kb * TC_BK;
          tma_load_2d(sA + s * C::A_BYTES, tmA, ka, mt * TC_BM, full + s);
          tma_load_2d(sB + s * C::B_BYTES, tmB, kw, nt * BN, full + s);
          ++issued;
          if (++s == C::STAGES) {
            s = 0;
            ph ^= 1;
          }
        }
      }
      if (!ok) {
        // drain: wait (bounded) for the copies this thread may still have in flight
        const uint64_t t0 = global_ns();
        for (int i = 0; i < C::STAGES && i < issued; ++i) {
          if (--s < 0) {
            s = C::STAGES - 1;
            ph ^= 1;
          }
          while (!mbar_try_wait(full + s, ph) && global_ns() - t0 < kWaitLimitNs) {
          }
        }
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      // ---------------- MMA issuer ----------------
      constexpr uint32_t idesc = idesc_bf16_f32(TC_BM, BN);
      int s = 0;
      uint32_t ph = 0;
      int acc = 0;
      uint32_t aph = 0;
      bool ok = true;
      for (int tile = blockIdx.x; tile < tiles && ok; tile += gridDim.x) {
        if (!mbar_wait(tempty + acc, aph ^ 1, abort_flag)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t dt = tmem_base + (uint32_t)(acc * BN);
        for (int kb = 0; kb < kit; ++kb) {
          if (!mbar_wait(full + s, ph, abort_flag)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t a0 = smem_u32(sA + s * C::A_BYTES);
          const uint32_t b0 = smem_u32(sB + s * C::B_BYTES);
#pragma unroll
          for (int k = 0; k < TC_BK / 16; ++k)
            mma_bf16(dt, sw128_desc(a0 + k * 32), sw128_desc(b0 + k * 32), idesc,
                     (kb | k) != 0 ? 1u : 0u);
          mma_commit(empty + s);
          if (++s == C::STAGES) {
            s = 0;
            ph ^= 1;
          }
        }
        if (!ok) break;
        mma_commit(tfull + acc);
        acc ^= 1;
        if (acc == 0) aph ^= 1;
      }
      // make sure every issued MMA has finished before TMEM is released
      mma_commit(drain);
      const uint64_t t0 = global_ns();
      while (!mbar_try_wait(drain, 0) && global_ns() - t0 < kWaitLimitNs) {
      }
    }
  } else {
    // ---------------- epilogue (warps 2..5 cover TMEM lane quarters 2,3,0,1) ----------------
    const int q = warp & 3;
    int acc = 0;
    uint32_t aph = 0;
    for (int tile = blockIdx.x; tile < tiles; tile += gridDim.x) {
      int pb, mt, nt;
      decode(tile, pb, mt, nt);
      const Epi& e = pb ? e1 : e0;
      bool ok = mbar_wait(tfull + acc, aph, abort_flag);
      if (!__all_sync(0xffffffffu, ok)) break;
      tc_fence_after();
      const int row = mt * TC_BM + q * 32 + lane;
      const uint32_t tb = tmem_base + (uint32_t)(acc * BN) + ((uint32_t)(q * 32) << 16);
      drain_accumulator<BN>(e, t, row, nt * BN, tb, vt_scratch + (warp - 2) * kVtScratchFloats);
      tc_fence_before();
      mbar_arrive(tempty + acc);
      acc ^= 1;
      if (acc == 0) aph ^= 1;
    }
  }
  __syncthreads();
  if (threadIdx.x == 0 && *abort_flag && err) atomicOr(err, 1);
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem_base, C::TMEM_COLS);
  }
}

template <int BN>
static cudaError_t launch_tc(const void* A0, long lda0, const void* W0, long ldw0, int M0,
                             const Epi& e0, const void* A1, long lda1, const void* W1, long ldw1,
                             int M1, const Epi& e1, int N, int K, int* err, cudaStream_t s,
                             int a_split) {
  using C = TcCfg<BN>;
  const uint64_t ka = (uint64_t)K * (a_split ? 2 : 1);
  CUtensorMap ta0, tb0, ta1, tb1;
  if (encode_tmap_2d_bf16(&ta0, A0, ka, (uint64_t)M0, (uint64_t)lda0 * 2, TC_BK, TC_BM) ||
      encode_tmap_2d_bf16(&tb0, W0, (uint64_t)K, (uint64_t)N, (uint64_t)ldw0 * 2, TC_BK, BN))
    return cudaErrorInvalidValue;
  if (M1 > 0) {
    if (encode_tmap_2d_bf16(&ta1, A1, ka, (uint64_t)M1, (uint64_t)lda1 * 2, TC_BK, TC_BM) ||
        encode_tmap_2d_bf16(&tb1, W1, (uint64_t)K, (uint64_t)N, (uint64_t)ldw1 * 2, TC_BK, BN))
      return cudaErrorInvalidValue;
  } else {
    ta1 = ta0;
    tb1 = tb0;
  }
  const int tiles = ((M0 + TC_BM - 1) / TC_BM + (M1 + TC_BM - 1) / TC_BM) * (N / BN);
  const int grid = std::min(tiles, num_sms());
  launch_kernel(gemm_tc_kernel<BN>, grid, 192, C::SMEM, s, ta0, tb0, ta1, tb1, e0, e1, M0, M1, N, K,
                a_split, tile_group_rows(M0, TC_BM, K, a_split),
                tile_group_rows(M1, TC_BM, K, a_split), err);
  return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// CTA-pair GEMM: clusters of two CTAs compute 256 x 256 tiles with cta_group::2 MMAs
// (M = 256, N = 256, K = 16 per instruction).  Each CTA stages its own 128 rows of A
// and 128 rows of W per k-block (32 KB instead of the single-CTA 128 x 256 tile's
// 48 KB), so every SM moves a third less shared-memory operand data per MMA cycle, the
// limit of the single-CTA kernel.  Roles as in gemm_tc_kernel: warp 0 of each CTA loads
// its halves (completion signalled on the even CTA's barrier), warp 1 of the even CTA
// issues the MMAs and multicasts their completion to both CTAs, warps 2..5 of each CTA
// drain its 128 accumulator rows.
// ---------------------------------------------------------------------------
constexpr int PR_BM = 256, PR_BN = 256, PR_STAGES = 6;
constexpr int PR_HALF_BYTES = 128 * TC_BK * 2;  // one CTA's A or W half-tile per k-block
constexpr int PR_STAGE_BYTES = 2 * PR_HALF_BYTES;
constexpr int PR_TMEM_COLS = 2 * PR_BN;         // double-buffered accumulator
constexpr int PR_SMEM = PR_STAGES * PR_STAGE_BYTES + 1024 + 256 + kVtScratchBytes;

__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(192, 1)
    gemm_pair_kernel(const __grid_constant__ CUtensorMap tmA0, const __grid_constant__ CUtensorMap tmB0,
                     const __grid_constant__ CUtensorMap tmA1, const __grid_constant__ CUtensorMap tmB1,
                     const __grid_constant__ Epi e0, const __grid_constant__ Epi e1, int M0, int M1,
                     int N, int K, int a_split, int g0, int g1, int* err) {
  grid_dep_sync();
  // both CTAs of a pair see the same flag, so they leave together
  if (epi_skip(e0.st, e0.flag_want)) return;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  uint8_t* sA = smem;
  uint8_t* sB = smem + PR_STAGES * PR_HALF_BYTES;
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + PR_STAGES * PR_STAGE_BYTES);
  uint64_t* empty = full + PR_STAGES;
  uint64_t* tfull = empty + PR_STAGES;
  uint64_t* tempty = tfull + 2;
  uint64_t* drain = tempty + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain + 1);
  float* vt_scratch = reinterpret_cast<float*>(smem + PR_STAGES * PR_STAGE_BYTES + 256);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
  const uint32_t rank = cluster_ctarank();
  const int pair = blockIdx.x >> 1, npairs = gridDim.x >> 1;
  const int num_m0 = (M0 + PR_BM - 1) / PR_BM, num_m1 = (M1 + PR_BM - 1) / PR_BM, num_n = N / PR_BN;
  const int tiles0 = num_m0 * num_n;
  auto decode = [&](int tile, int& pb, int& mt, int& nt) {
    if (tile < tiles0) {
      pb = 0;
      raster(tile, num_m0, num_n, g0, mt, nt);
    } else {
      pb = 1;
      raster(tile - tiles0, num_m1, num_n, g1, mt, nt);
    }
  };
  const int tiles = tiles0 + num_m1 * num_n, kit = (a_split ? 2 : 1) * (K / TC_BK);
  const int t = epi_step(e0);

  if (threadIdx.x == 0) {
    for (int s = 0; s < PR_STAGES; ++s) {
      mbar_init(full + s, 1);   // even CTA: its producer's expect_tx; both CTAs' bytes
      mbar_init(empty + s, 1);  // both CTAs: one multicast commit per consumed stage
    }
    mbar_init(tfull, 1);
    mbar_init(tfull + 1, 1);
    mbar_init(tempty, 256);     // even CTA: every epilogue thread of both CTAs
    mbar_init(tempty + 1, 256);
    mbar_init(drain, 1);
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == 0 && lane == 0) {
    tma_prefetch_desc(&tmA0);
    tma_prefetch_desc(&tmB0);
    if (M1 > 0) {
      tma_prefetch_desc(&tmA1);
      tma_prefetch_desc(&tmB1);
    }
  }
  __syncwarp();
  if (warp == 1) {
    tmem_alloc_pair(tmem_slot, PR_TMEM_COLS);
    tmem_relinquish_pair();
  }
  tc_fence_before();
  __syncwarp();
  cluster_sync_all();  // barriers of both CTAs initialised, tensor memory allocated
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;

  if (warp == 0) {
    if (lane == 0) {
      // ---------------- TMA producer (both CTAs: their own halves) ----------------
      int s = 0;
      uint32_t ph = 0;
      long issued = 0;
      bool ok = true;
      for (int tile = pair; tile < tiles && ok; tile += npairs) {
        int pb, mt, nt;
        decode(tile, pb, mt, nt);
        const CUtensorMap* tmA = pb ? &tmA1 : &tmA0;
        const CUtensorMap* tmB = pb ? &tmB1 : &tmB0;
        for (int kb = 0; kb < kit; ++kb) {
          if (!mbar_wait(empty + s, ph ^ 1, abort_flag)) {
            ok = false;
            break;
          }
          if (rank == 0) mbar_arrive_expect_tx(full + s, 2 * PR_STAGE_BYTES);
          const uint32_t fb = mapa_shared(smem_u32(full + s), 0);
          const int ka = a_split ? (kb & 1) * K + (kb >> 1) * TC_BK : kb * TC_BK;
          const int kw = a_split ? (kb >> 1) * TC_BK : kb * TC_BK;
          tma_load_2d_pair(sA + s * PR_HALF_BYTES, tmA, ka, mt * PR_BM + (int)rank * 128, fb);
          tma_load_2d_pair(sB + s * PR_HALF_BYTES, tmB, kw, nt * PR_BN + (int)rank * 128, fb);
          ++issued;
          if (++s == PR_STAGES) {
            s = 0;
            ph ^= 1;
          }
        }
      }
      if (!ok && rank == 0) {
        // drain (bounded): both CTAs' copies in flight complete on this CTA's barriers
        const uint64_t t0 = global_ns();
        for (int i = 0; i < PR_STAGES && i < issued; ++i) {
          if (--s < 0) {
            s = PR_STAGES - 1;
            ph ^= 1;
          }
          while (!mbar_try_wait(full + s, ph) && global_ns() - t0 < kWaitLimitNs) {
          }
        }
      }
    }
  } else if (warp == 1) {
    if (lane == 0 && rank == 0) {
      // ---------------- MMA issuer (even CTA) ----------------
      constexpr uint32_t idesc = idesc_bf16_f32(PR_BM, PR_BN);
      int s = 0;
      uint32_t ph = 0;
      int acc = 0;
      uint32_t aph = 0;
      bool ok = true;
      for (int tile = pair; tile < tiles && ok; tile += npairs) {
        if (!mbar_wait(tempty + acc, aph ^ 1, abort_flag)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t dt = tmem_base + (uint32_t)(acc * PR_BN);
        for (int kb = 0; kb < kit; ++kb) {
          if (!mbar_wait(full + s, ph, abort_flag)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t a0 = smem_u32(sA + s * PR_HALF_BYTES);
          const uint32_t b0 = smem_u32(sB + s * PR_HALF_BYTES);
#pragma unroll
          for (int k = 0; k < TC_BK / 16; ++k)
            mma_bf16_pair(dt, sw128_desc(a0 + k * 32), sw128_desc(b0 + k * 32), idesc,
                          (kb | k) != 0 ? 1u : 0u);
          mma_commit_pair(empty + s, 3);
          if (++s == PR_STAGES) {
            s = 0;
            ph ^= 1;
          }
        }
        if (!ok) break;
        mma_commit_pair(tfull + acc, 3);
        acc ^= 1;
        if (acc == 0) aph ^= 1;
      }
      // every issued MMA has finished before tensor memory is released
      mma_commit_pair(drain, 1);
      const uint64_t t0 = global_ns();
      while (!mbar_try_wait(drain, 0) && global_ns() - t0 < kWaitLimitNs) {
      }
    }
  } else {
    // ---------------- epilogue (both CTAs: their 128 rows of each tile) ----------------
    const int q = warp & 3;
    int acc = 0;
    uint32_t aph = 0;
    const uint32_t te_remote = mapa_shared(smem_u32(tempty), 0);
    for (int tile = pair; tile < tiles; tile += npairs) {
      int pb, mt, nt;
      decode(tile, pb, mt, nt);
      const Epi& e = pb ? e1 : e0;
      bool ok = mbar_wait(tfull + acc, aph, abort_flag);
      if (!__all_sync(0xffffffffu, ok)) break;
      tc_fence_after();
      const int row = mt * PR_BM + (int)rank * 128 + q * 32 + lane;
      const uint32_t tb = tmem_base + (uint32_t)(acc * PR_BN) + ((uint32_t)(q * 32) << 16);
      drain_accumulator<PR_BN>(e, t, row, nt * PR_BN, tb, vt_scratch + (warp - 2) * kVtScratchFloats);
      tc_fence_before();
      if (rank == 0)
        mbar_arrive(tempty + acc);
      else
        mbar_arrive_remote(te_remote + (uint32_t)(acc * sizeof(uint64_t)));
      acc ^= 1;
      if (acc == 0) aph ^= 1;
    }
  }
  tc_fence_before();
  __syncwarp();
  cluster_sync_all();  // no CTA of the pair still uses the pair's tensor memory
  if (threadIdx.x == 0 && *abort_flag && err) atomicOr(err, 1);
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc_pair(tmem_base, PR_TMEM_COLS);
  }
}

// Tiles of the pair kernel for a launch of one or two problems; it is used when N is a
// multiple of 256 and there are at least as many 256 x 256 tiles as CTA pairs.
static int pair_tiles(int M0, int M1, int N) {
  return ((M0 + PR_BM - 1) / PR_BM + (M1 + PR_BM - 1) / PR_BM) * (N / PR_BN);
}

static cudaError_t launch_pair(const void* A0, long lda0, const void* W0, long ldw0, int M0,
                               const Epi& e0, const void* A1, long lda1, const void* W1, long ldw1,
                               int M1, const Epi& e1, int N, int K, int* err, cudaStream_t s,
                               int a_split) {
  const uint64_t ka = (uint64_t)K * (a_split ? 2 : 1);
  CUtensorMap ta0, tb0, ta1, tb1;
  if (encode_tmap_2d_bf16(&ta0, A0, ka, (uint64_t)M0, (uint64_t)lda0 * 2, TC_BK, 128) ||
      encode_tmap_2d_bf16(&tb0, W0, (uint64_t)K, (uint64_t)N, (uint64_t)ldw0 * 2, TC_BK, 128))
    return cudaErrorInvalidValue;
  if (M1 > 0) {
    if (encode_tmap_2d_bf16(&ta1, A1, ka, (uint64_t)M1, (uint64_t)lda1 * 2, TC_BK, 128) ||
        encode_tmap_2d_bf16(&tb1, W1, (uint64_t)K, (uint64_t)N, (uint64_t)ldw1 * 2, TC_BK, 128))
      return cudaErrorInvalidValue;
  } else {
    ta1 = ta0;
    tb1 = tb0;
  }
  const int pairs = std::min(pair_tiles(M0, M1, N), num_sms() / 2);
  launch_kernel(gemm_pair_kernel, 2 * pairs, 192, PR_SMEM, s, ta0, tb0, ta1, tb1, e0, e1, M0, M1, N,
                K, a_split, tile_group_rows(M0, PR_BM, K, a_split),
                tile_group_rows(M1, PR_BM, K, a_split), err);
  return cudaGetLastError();
}

int gemm_uses_pair(int M0, int M1, int N) {
  return N % PR_BN == 0 && num_sms() >= 2 && pair_tiles(M0, M1, N) >= num_sms() / 2;
}

cudaError_t attention_tc_init();

cudaError_t kernels_init() {
  cudaError_t r = cudaFuncSetAttribute(gemm_tc_kernel<256>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       TcCfg<256>::SMEM);
  if (r == cudaSuccess)
    r = cudaFuncSetAttribute(gemm_tc_kernel<128>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             TcCfg<128>::SMEM);
  if (r == cudaSuccess)
    r = cudaFuncSetAttribute(gemm_tc_kernel<64>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             TcCfg<64>::SMEM);
  if (r == cudaSuccess)
    r = cudaFuncSetAttribute(gemm_pair_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, PR_SMEM);
  if (r == cudaSuccess) r = attention_tc_init();
  num_sms();
  return r;
}

int gemm_tc_supported(int M, int N, int K, long lda, long ldw) {
  if (M <= 0 || K <= 0 || K % TC_BK != 0 || N % 64 != 0) return 0;
  if (lda % 8 != 0 || ldw % 8 != 0) return 0;
  return get_encode_fn() != nullptr;
}

// tensor-core launch of one or two problems (M1 = 0: one); picks the widest tile that
// still gives every SM at least one tile
static cudaError_t gemm_tc2(const void* A0, long lda0, const void* W0, long ldw0, int M0,
                            const Epi& e0, const void* A1, long lda1, const void* W1, long ldw1,
                            int M1, const Epi& e1, int N, int K, int* err, cudaStream_t s,
                            int a_split) {
  const uintptr_t ptrs = reinterpret_cast<uintptr_t>(A0) | reinterpret_cast<uintptr_t>(W0) |
                         (M1 > 0 ? (reinterpret_cast<uintptr_t>(A1) | reinterpret_cast<uintptr_t>(W1)) : 0);
  if ((ptrs & 15) || !gemm_tc_supported(M0, N, K, lda0, ldw0) ||
      (M1 > 0 && !gemm_tc_supported(M1, N, K, lda1, ldw1)))
    return cudaErrorNotSupported;
  if (a_split && (lda0 < 2L * K || (M1 > 0 && lda1 < 2L * K))) return cudaErrorInvalidValue;
  const int ns = num_sms();
  const int mt = (M0 + TC_BM - 1) / TC_BM + (M1 + TC_BM - 1) / TC_BM;
  // QK-norm epilogues need whole heads in a tile: BN a multiple of dh
  const bool qkn = e0.qn_q || (M1 > 0 && e1.qn_q);
  const int min_bn = qkn ? e0.dh : 64;
  if (qkn && (e0.dh % 32 || (M1 > 0 && e1.dh != e0.dh) || min_bn > 256)) return cudaErrorNotSupported;
  if (gemm_uses_pair(M0, M1 > 0 ? M1 : 0, N))
    return launch_pair(A0, lda0, W0, ldw0, M0, e0, A1, lda1, W1, ldw1, M1 > 0 ? M1 : 0, e1, N, K, err, s,
                       a_split);
  if (N % 256 == 0 && (mt * (N / 256) >= ns || min_bn > 128))
    return launch_tc<256>(A0, lda0, W0, ldw0, M0, e0, A1, lda1, W1, ldw1, M1, e1, N, K, err, s, a_split);
  if (min_bn > 128) return cudaErrorNotSupported;
  if (N % 128 == 0 && (mt * (N / 128) >= ns || min_bn > 64))
    return launch_tc<128>(A0, lda0, W0, ldw0, M0, e0, A1, lda1, W1, ldw1, M1, e1, N, K, err, s, a_split);
  if (min_bn > 64) return cudaErrorNotSupported;
  return launch_tc<64>(A0, lda0, W0, ldw0, M0, e0, A1, lda1, W1, ldw1, M1, e1, N, K, err, s, a_split);
}

cudaError_t gemm2(const void* A0, long lda0, const void* W0, long ldw0, int M0, const Epi& epi0,
                  const void* A1, long lda1, const void* W1, long ldw1, int M1, const Epi& epi1,
                  int N, int K, int* err, cudaStream_t s) {
  if (N <= 0 || (M0 <= 0 && M1 <= 0)) return cudaSuccess;
  Epi e0 = epi0, e1 = epi1;
  e0.M = M0;
  e0.N = N;
  e1.M = M1;
  e1.N = N;
  if (M0 <= 0) return gemm_tc2(A1, lda1, W1, ldw1, M1, e1, nullptr, 0, nullptr, 0, 0, e1, N, K, err, s, 0);
  return gemm_tc2(A0, lda0, W0, ldw0, M0, e0, A1, lda1, W1, ldw1, M1 > 0 ? M1 : 0, e1, N, K, err, s, 0);
}

cudaError_t gemm(const void* A, long lda, const void* W, long ldw, int M, int N, int K,
                 int in_bf16, const Epi& epi_in, int* err, cudaStream_t s, int force_simt,
                 int a_split) {
  if (M <= 0 || N <= 0) return cudaSuccess;
  Epi e = epi_in;
  e.M = M;
  e.N = N;
  if (in_bf16 && !force_simt) {
    // bf16 operands always take the tensor-core path; a shape or pointer it cannot
    // tile is an error, never a silent switch to the CUDA-core kernel
    return gemm_tc2(A, lda, W, ldw, M, e, nullptr, 0, nullptr, 0, 0, e, N, K, err, s, a_split);
  }
  if (a_split) return cudaErrorInvalidValue;
  if (N % 4 != 0) return cudaErrorInvalidValue;
  dim3 grid((N + 63) / 64, (M + 63) / 64);
  if (in_bf16)
    launch_kernel(gemm_simt_kernel<__nv_bfloat16>, grid, 256, 0, s,
                  reinterpret_cast<const __nv_bfloat16*>(A), lda,
                  reinterpret_cast<const __nv_bfloat16*>(W), ldw, M, N, K, e);
  else
    launch_kernel(gemm_simt_kernel<float>, grid, 256, 0, s, reinterpret_cast<const float*>(A), lda,
                  reinterpret_cast<const float*>(W), ldw, M, N, K, e);
  return cudaGetLastError();
}

}  // namespace bag
