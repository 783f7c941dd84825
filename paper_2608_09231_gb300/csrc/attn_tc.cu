// Joint attention on the 5th-generation tensor cores (head_dim 128, bf16 operands).
//
// One CTA owns 128 query rows of one head and walks the keys in tiles of 128:
//   warp 0      TMA producer: Q once, then K and V^T tiles into a 2-stage ring
//   warp 1      MMA issuer:   S_j = Q K_j^T into one of two TMEM buffers, then
//                             O += P_{j-1} V_{j-1} (P from shared memory), so the tensor
//                             core computes S_{j+1} while the softmax works on S_j
//   warps 2..5  softmax:      thread = query row; S row from TMEM, running max/sum in
//                             the exp2 domain, P = exp2(s - m) as bf16 into shared
//                             memory (128-byte swizzle, K-major for the PV MMA).
// O lives in TMEM for the whole key loop.  The running max is only moved (and O
// rescaled in TMEM) when a tile's max exceeds it by more than 8 in log2 units, so P
// stays <= 2^8 and the rescale is rare; the final division by the row sum uses the
// same max, so the result is the exact softmax up to rounding.
// V arrives transposed per head ([head][dh][token]) from the QKV projection's epilogue,
// which makes it a K-major B operand like every other tile here.
#include <cmath>

#include "common.cuh"
#include "epilogue.cuh"
#include "kernels.h"

namespace bag {

namespace {
constexpr int AT_M = 128, AT_N = 128, AT_D = 128;
constexpr int AT_CHUNK = 128 * 64 * 2;  // 128 rows x 64 bf16 = one 128-byte-swizzle column
constexpr int AT_TILE = 2 * AT_CHUNK;   // 128 x 128 bf16
constexpr int AT_STAGES = 2;
constexpr int AT_OFF_Q = 0;
constexpr int AT_OFF_KV = AT_TILE;                              // stage s: K, then V^T
constexpr int AT_OFF_P = AT_OFF_KV + AT_STAGES * 2 * AT_TILE;
constexpr int AT_OFF_BAR = AT_OFF_P + AT_TILE;
constexpr int AT_SMEM = AT_OFF_BAR + 256 + 1024;
constexpr int AT_TMEM_COLS = 512;  // S0 [0,128), S1 [128,256), O [256,384)

struct AttnTcParams {
  int nq, nk;
  void* o;
  long ldo;
  float scale_log2;
  const DevState* st;
  int flag_want;
  int* err;
};

BAG_DEV float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// byte offset of 16-byte unit u (0..15, 8 bf16 each) of row r in a 128 x 128 bf16 tile
// stored as two 128-byte-swizzled K-major columns
BAG_DEV uint32_t sw_off(int r, int u) {
  return (uint32_t)((u >> 3) * AT_CHUNK + (r >> 3) * 1024 + (r & 7) * 128 + (((u & 7) ^ (r & 7)) << 4));
}
}  // namespace

__global__ void __launch_bounds__(192, 1)
    attn_tc_kernel(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
                   const __grid_constant__ CUtensorMap tmV, const AttnTcParams p) {
  if (epi_skip(p.st, p.flag_want)) return;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  uint8_t* sQ = smem + AT_OFF_Q;
  uint8_t* sKV = smem + AT_OFF_KV;
  uint8_t* sP = smem + AT_OFF_P;
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + AT_OFF_BAR);
  uint64_t* q_full = bars + 0;
  uint64_t* kv_full = bars + 1;   // [2]
  uint64_t* kv_empty = bars + 3;  // [2]
  uint64_t* s_full = bars + 5;    // [2]
  uint64_t* s_free = bars + 7;    // [2]
  uint64_t* p_full = bars + 9;
  uint64_t* o_done = bars + 10;
  uint64_t* drain = bars + 11;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 12);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
  const int head = blockIdx.y, q0 = blockIdx.x * AT_M;
  const int nkb = (p.nk + AT_N - 1) / AT_N;

  if (threadIdx.x == 0) {
    mbar_init(q_full, 1);
    for (int i = 0; i < 2; ++i) {
      mbar_init(kv_full + i, 1);
      mbar_init(kv_empty + i, 1);
      mbar_init(s_full + i, 1);
      mbar_init(s_free + i, 128);
    }
    mbar_init(p_full, 128);
    mbar_init(o_done, 1);
    mbar_init(drain, 1);
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == 0 && lane == 0) {
    tma_prefetch_desc(&tmQ);
    tma_prefetch_desc(&tmK);
    tma_prefetch_desc(&tmV);
  }
  if (warp == 1) {
    tmem_alloc(tmem_slot, AT_TMEM_COLS);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (warp == 0) {
    if (lane == 0) {
      // ---------------- TMA producer ----------------
      mbar_arrive_expect_tx(q_full, AT_TILE);
      tma_load_2d(sQ, &tmQ, head * AT_D, q0, q_full);
      tma_load_2d(sQ + AT_CHUNK, &tmQ, head * AT_D + 64, q0, q_full);
      int issued = 0;
      bool ok = true;
      for (int j = 0; j < nkb; ++j) {
        const int s = j % AT_STAGES;
        if (!mbar_wait(kv_empty + s, ((j / AT_STAGES) & 1) ^ 1, abort_flag)) {
          ok = false;
          break;
        }
        uint8_t* k = sKV + s * 2 * AT_TILE;
        uint8_t* v = k + AT_TILE;
        mbar_arrive_expect_tx(kv_full + s, 2 * AT_TILE);
        tma_load_2d(k, &tmK, head * AT_D, j * AT_N, kv_full + s);
        tma_load_2d(k + AT_CHUNK, &tmK, head * AT_D + 64, j * AT_N, kv_full + s);
        tma_load_2d(v, &tmV, j * AT_N, head * AT_D, kv_full + s);
        tma_load_2d(v + AT_CHUNK, &tmV, j * AT_N + 64, head * AT_D, kv_full + s);
        ++issued;
      }
      if (!ok) {
        // wait (bounded) for copies still in flight before the CTA may exit
        const uint64_t t0 = global_ns();
        while (!mbar_try_wait(q_full, 0) && global_ns() - t0 < kWaitLimitNs) {
        }
        for (int j = (issued > AT_STAGES ? issued - AT_STAGES : 0); j < issued; ++j)
          while (!mbar_try_wait(kv_full + j % AT_STAGES, (j / AT_STAGES) & 1) &&
                 global_ns() - t0 < kWaitLimitNs) {
          }
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      // ---------------- MMA issuer ----------------
      constexpr uint32_t idesc = idesc_bf16_f32(AT_M, AT_N);
      bool ok = mbar_wait(q_full, 0, abort_flag);
      tc_fence_after();
      const uint32_t q_addr = smem_u32(sQ), p_addr = smem_u32(sP);
      auto issue_pv = [&](int i) -> bool {
        if (!mbar_wait(p_full, i & 1, abort_flag)) return false;
        tc_fence_after();
        const uint32_t v_addr = smem_u32(sKV + (i % AT_STAGES) * 2 * AT_TILE + AT_TILE);
#pragma unroll
        for (int kk = 0; kk < AT_N / 16; ++kk) {
          const uint32_t off = (kk >> 2) * AT_CHUNK + (kk & 3) * 32;
          mma_bf16(tmem + 256, sw128_desc(p_addr + off), sw128_desc(v_addr + off), idesc,
                   (i > 0 || kk > 0) ? 1u : 0u);
        }
        mma_commit(o_done);
        mma_commit(kv_empty + i % AT_STAGES);
        return true;
      };
      for (int j = 0; j < nkb && ok; ++j) {
        const int s = j % AT_STAGES, b = j & 1;
        if (!mbar_wait(kv_full + s, (j / AT_STAGES) & 1, abort_flag)) {
          ok = false;
          break;
        }
        if (j >= 2 && !mbar_wait(s_free + b, ((j - 2) >> 1) & 1, abort_flag)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t k_addr = smem_u32(sKV + s * 2 * AT_TILE);
#pragma unroll
        for (int kk = 0; kk < AT_D / 16; ++kk) {
          const uint32_t off = (kk >> 2) * AT_CHUNK + (kk & 3) * 32;
          mma_bf16(tmem + b * 128, sw128_desc(q_addr + off), sw128_desc(k_addr + off), idesc,
                   kk > 0 ? 1u : 0u);
        }
        mma_commit(s_full + b);
        if (j >= 1 && !issue_pv(j - 1)) ok = false;
      }
      if (ok) issue_pv(nkb - 1);
      mma_commit(drain);
      const uint64_t t0 = global_ns();
      while (!mbar_try_wait(drain, 0) && global_ns() - t0 < kWaitLimitNs) {
      }
    }
  } else {
    // ---------------- softmax warpgroup ----------------
    const int quad = warp & 3;
    const int row = quad * 32 + lane;
    const uint32_t lane_base = (uint32_t)(quad * 32) << 16;
    float m_use = -INFINITY, l = 0.f;
    bool ok = true;
    for (int j = 0; j < nkb; ++j) {
      const int b = j & 1;
      bool w = mbar_wait(s_full + b, (j >> 1) & 1, abort_flag);
      if (!__all_sync(0xffffffffu, w)) {
        ok = false;
        break;
      }
      tc_fence_after();
      float s[AT_N];
#pragma unroll
      for (int c = 0; c < AT_N / 32; ++c) tmem_ld32(tmem + lane_base + b * 128 + c * 32, s + c * 32);
      tc_fence_before();
      mbar_arrive(s_free + b);
      const int kvalid = p.nk - j * AT_N;
      if (kvalid < AT_N) {
#pragma unroll
        for (int i = 0; i < AT_N; ++i)
          if (i >= kvalid) s[i] = -INFINITY;
      }
      float mx = s[0];
#pragma unroll
      for (int i = 1; i < AT_N; ++i) mx = fmaxf(mx, s[i]);
      const float mx2 = mx * p.scale_log2;
      float alpha = 1.f;
      if (mx2 > m_use + 8.f) {
        alpha = ex2(m_use - mx2);
        m_use = mx2;
        l *= alpha;
      }
      const bool resc = __any_sync(0xffffffffu, alpha != 1.f) && j > 0;
      uint32_t pk[AT_N / 2];
      float ls = 0.f;
#pragma unroll
      for (int i = 0; i < AT_N; i += 2) {
        const float a0 = ex2(fmaf(s[i], p.scale_log2, -m_use));
        const float a1 = ex2(fmaf(s[i + 1], p.scale_log2, -m_use));
        ls += a0 + a1;
        pk[i / 2] = pack_bf16x2(a0, a1);
      }
      l += ls;
      if (j >= 1) {
        w = mbar_wait(o_done, (j - 1) & 1, abort_flag);
        if (!__all_sync(0xffffffffu, w)) {
          ok = false;
          break;
        }
        tc_fence_after();
      }
      if (resc) {
#pragma unroll 1
        for (int c = 0; c < AT_D / 32; ++c) {
          float o[32];
          tmem_ld32(tmem + lane_base + 256 + c * 32, o);
#pragma unroll
          for (int i = 0; i < 32; ++i) o[i] *= alpha;
          tmem_st32(tmem + lane_base + 256 + c * 32, o);
        }
        tmem_st_wait();
      }
      const uint32_t pbase = smem_u32(sP);
#pragma unroll
      for (int u = 0; u < AT_N / 8; ++u) {
        asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(pbase + sw_off(row, u)),
                     "r"(pk[4 * u]), "r"(pk[4 * u + 1]), "r"(pk[4 * u + 2]), "r"(pk[4 * u + 3])
                     : "memory");
      }
      fence_proxy_async_smem();
      tc_fence_before();
      mbar_arrive(p_full);
    }
    if (ok) {
      bool w = mbar_wait(o_done, (nkb - 1) & 1, abort_flag);
      if (__all_sync(0xffffffffu, w)) {
        tc_fence_after();
        const float inv = 1.f / l;
        const int q = q0 + row;
        __nv_bfloat16* orow = reinterpret_cast<__nv_bfloat16*>(p.o) + (long)q * p.ldo + head * AT_D;
#pragma unroll 1
        for (int c = 0; c < AT_D / 32; ++c) {
          float o[32];
          tmem_ld32(tmem + lane_base + 256 + c * 32, o);
#pragma unroll
          for (int i = 0; i < 32; ++i) o[i] *= inv;
          if (q < p.nq) store_vals<32>(orow + c * 32, 0, o, 1);
        }
      }
    }
  }
  __syncthreads();
  if (threadIdx.x == 0 && *abort_flag && p.err) atomicOr(p.err, 1);
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, AT_TMEM_COLS);
  }
}

cudaError_t attention_tc_init() {
  return cudaFuncSetAttribute(attn_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, AT_SMEM);
}

int attention_tc_supported(const AttnArgs& a) {
  if (!a.bf16 || a.dh != AT_D || a.v_mode != 1) return 0;
  if (a.ldq % 8 || a.ldk % 8 || a.vpad % 8 || a.ldo % 8) return 0;
  if ((reinterpret_cast<uintptr_t>(a.q) | reinterpret_cast<uintptr_t>(a.k) |
       reinterpret_cast<uintptr_t>(a.v) | reinterpret_cast<uintptr_t>(a.o)) & 15)
    return 0;
  return a.nq > 0 && a.nk > 0 && a.vpad >= a.nk;
}

cudaError_t attention_tc(const AttnArgs& a, int* err, cudaStream_t s) {
  CUtensorMap tq, tk, tv;
  const uint64_t width = (uint64_t)a.heads * AT_D;
  if (encode_tmap_2d_bf16(&tq, a.q, width, (uint64_t)a.nq, (uint64_t)a.ldq * 2, 64, AT_M) ||
      encode_tmap_2d_bf16(&tk, a.k, width, (uint64_t)a.nk, (uint64_t)a.ldk * 2, 64, AT_N) ||
      encode_tmap_2d_bf16(&tv, a.v, (uint64_t)a.nk, width, (uint64_t)a.vpad * 2, 64, AT_D))
    return cudaErrorInvalidValue;
  AttnTcParams p;
  p.nq = a.nq;
  p.nk = a.nk;
  p.o = a.o;
  p.ldo = a.ldo;
  p.scale_log2 = (float)(1.4426950408889634 / std::sqrt((double)AT_D));
  p.st = a.st;
  p.flag_want = a.flag_want;
  p.err = err;
  dim3 grid((a.nq + AT_M - 1) / AT_M, a.heads);
  attn_tc_kernel<<<grid, 192, AT_SMEM, s>>>(tq, tk, tv, p);
  return cudaGetLastError();
}

}  // namespace bag
