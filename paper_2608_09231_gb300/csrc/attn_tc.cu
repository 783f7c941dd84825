// Joint attention on the 5th-generation tensor cores (head_dim 128, 16-bit operands).
//
// One CTA owns two 128-row query tiles (A and B) of one head and walks the keys in
// tiles of 128:
//   warp 0      TMA producer: both Q tiles once, then K and V^T tiles into a 2-stage ring
//   warp 1      MMA issuer, ping-pong between the tiles:
//                 S_A,0  S_B,0 | PV_A,j  S_A,j+1 | PV_B,j  S_B,j+1 | ...
//               so the tensor core computes one tile's products while the other tile's
//               softmax runs
//   warps 2..5  softmax of tile A, warps 6..9 softmax of tile B: thread = query row; S
//               row read from TMEM into registers in one round trip, P = exp2(s - m)
//               packed to 16 bits and written back into TMEM over the S columns.
// The PV product takes P straight from TMEM as its A operand, so P never touches
// shared memory; shared memory only feeds Q, K and V^T.  O stays in TMEM for the whole
// key loop.  The running max only moves (and O is rescaled in TMEM) when a tile's max
// exceeds it by more than 8 in log2 units, so P <= 2^8; the final division by the row
// sum uses the same max, which makes the result the exact softmax up to rounding.
// V arrives transposed per head ([head][dh][token]) from the QKV projection's epilogue,
// which makes it a K-major B operand.
// Operands are bf16 or fp16 (F16): q, k, v and P all of that type (an MMA's A and B share
// one type).  The sampling path uses fp16: its 11-bit significand rounds q and k, whose
// errors the softmax exponent amplifies, eight times more finely than bf16, and P stays
// within fp16's range because the lazy maximum bounds it by 2^8.
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
constexpr int AT_OFF_Q = 0;                                     // Q_A, Q_B
constexpr int AT_OFF_KV = 2 * AT_TILE;                          // stage s: K, then V^T
constexpr int AT_OFF_BAR = AT_OFF_KV + AT_STAGES * 2 * AT_TILE;
constexpr int AT_SMEM = AT_OFF_BAR + 256 + 1024;
constexpr int AT_TMEM_COLS = 512;  // S_A [0,128) S_B [128,256) O_A [256,384) O_B [384,512)
constexpr int AT_THREADS = 320;

struct AttnTcParams {
  int nq, nk;
  void* o;
  long ldo;
  void* o2;     // rows >= o_split are written to o2 (same row index and stride)
  int o_split;
  // branch blockIdx.z: q / k row offsets, V^T row offset (per branch block), outputs
  int br_q_rows, br_k_rows, br_v_rows;
  void* o_b1;
  void* o2_b1;
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

// Three-input maximum and packed two-lane fp32 FMA / add (one instruction each for two
// elements of the S row, halving the softmax's issue slots for these steps).
BAG_DEV float max3(float a, float b, float c) {
  float d;
  asm("max.f32 %0, %1, %2, %3;" : "=f"(d) : "f"(a), "f"(b), "f"(c));
  return d;
}
BAG_DEV void fma2(float& d0, float& d1, float a0, float a1, float b, float c) {
  asm("{\n\t.reg .b64 ra, rb, rc, rd;\n\t"
      "mov.b64 ra, {%2, %3};\n\tmov.b64 rb, {%4, %4};\n\tmov.b64 rc, {%5, %5};\n\t"
      "fma.rn.f32x2 rd, ra, rb, rc;\n\tmov.b64 {%0, %1}, rd;\n\t}"
      : "=f"(d0), "=f"(d1)
      : "f"(a0), "f"(a1), "f"(b), "f"(c));
}
BAG_DEV void add2(float& d0, float& d1, float a0, float a1) {
  asm("{\n\t.reg .b64 ra, rd;\n\t"
      "mov.b64 ra, {%2, %3};\n\tmov.b64 rd, {%0, %1};\n\t"
      "add.rn.f32x2 rd, rd, ra;\n\tmov.b64 {%0, %1}, rd;\n\t}"
      : "+f"(d0), "+f"(d1)
      : "f"(a0), "f"(a1));
}

// 32 consecutive 32-bit TMEM columns of this thread's lane, without the wait (the caller
// issues tcgen05.wait::ld once for several loads)
BAG_DEV void tmem_ld32_nowait(uint32_t taddr, uint32_t* r) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
      "{%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, "
      "%16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31}, "
      "[%32];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
        "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]),
        "=r"(r[13]), "=r"(r[14]), "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]),
        "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]),
        "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]),
        "=r"(r[31])
      : "r"(taddr));
}

BAG_DEV void tmem_ld_wait() { asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory"); }

// 16 consecutive 32-bit TMEM columns of this thread's lane
BAG_DEV void tmem_st16(uint32_t taddr, const uint32_t* v) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], "
      "{%1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, %16};" ::"r"(taddr),
      "r"(v[0]), "r"(v[1]), "r"(v[2]), "r"(v[3]), "r"(v[4]), "r"(v[5]), "r"(v[6]), "r"(v[7]),
      "r"(v[8]), "r"(v[9]), "r"(v[10]), "r"(v[11]), "r"(v[12]), "r"(v[13]), "r"(v[14]),
      "r"(v[15])
      : "memory");
}

// D (TMEM) += A (TMEM, 16-bit elements packed two per column) * B (shared memory)
BAG_DEV void mma_bf16_ts(uint32_t d_tmem, uint32_t a_tmem, uint64_t bdesc, uint32_t idesc,
                         uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n\t}" ::"r"(d_tmem),
      "r"(a_tmem), "l"(bdesc), "r"(idesc), "r"(accumulate)
      : "memory");
}
}  // namespace

template <bool F16>
__global__ void __launch_bounds__(AT_THREADS, 1)
    attn_tc_kernel(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
                   const __grid_constant__ CUtensorMap tmV, const AttnTcParams p) {
  grid_dep_sync();
  if (epi_skip(p.st, p.flag_want)) return;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  uint8_t* sQ = smem + AT_OFF_Q;
  uint8_t* sKV = smem + AT_OFF_KV;
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + AT_OFF_BAR);
  uint64_t* q_full = bars + 0;
  uint64_t* kv_full = bars + 1;   // [2]
  uint64_t* kv_empty = bars + 3;  // [2]
  uint64_t* s_full = bars + 5;    // [2] per query tile
  uint64_t* p_full = bars + 7;    // [2]
  uint64_t* o_done = bars + 9;    // [2]
  uint64_t* drain = bars + 11;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 12);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
  const int head = blockIdx.y, q0 = blockIdx.x * 2 * AT_M;
  const int br = blockIdx.z;  // guidance branch (0 unless two branches share the launch)
  const int qr0 = q0 + br * p.br_q_rows, kr0 = br * p.br_k_rows, vr0 = br * p.br_v_rows;
  const int nkb = (p.nk + AT_N - 1) / AT_N;

  if (threadIdx.x == 0) {
    mbar_init(q_full, 1);
    for (int i = 0; i < 2; ++i) {
      mbar_init(kv_full + i, 1);
      mbar_init(kv_empty + i, 1);
      mbar_init(s_full + i, 1);
      mbar_init(p_full + i, 128);
      mbar_init(o_done + i, 1);
    }
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
      mbar_arrive_expect_tx(q_full, 2 * AT_TILE);
      for (int x = 0; x < 2; ++x) {
        tma_load_2d(sQ + x * AT_TILE, &tmQ, head * AT_D, qr0 + x * AT_M, q_full);
        tma_load_2d(sQ + x * AT_TILE + AT_CHUNK, &tmQ, head * AT_D + 64, qr0 + x * AT_M, q_full);
      }
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
        tma_load_2d(k, &tmK, head * AT_D, kr0 + j * AT_N, kv_full + s);
        tma_load_2d(k + AT_CHUNK, &tmK, head * AT_D + 64, kr0 + j * AT_N, kv_full + s);
        tma_load_2d(v, &tmV, j * AT_N, vr0 + head * AT_D, kv_full + s);
        tma_load_2d(v + AT_CHUNK, &tmV, j * AT_N + 64, vr0 + head * AT_D, kv_full + s);
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
      constexpr uint32_t idesc = F16 ? idesc_f16_f32(AT_M, AT_N) : idesc_bf16_f32(AT_M, AT_N);
      const uint32_t q_addr = smem_u32(sQ);
      auto issue_s = [&](int x, int j) {
        const uint32_t qa = q_addr + x * AT_TILE;
        const uint32_t ka = smem_u32(sKV + (j % AT_STAGES) * 2 * AT_TILE);
#pragma unroll
        for (int kk = 0; kk < AT_D / 16; ++kk) {
          const uint32_t off = (kk >> 2) * AT_CHUNK + (kk & 3) * 32;
          mma_bf16(tmem + x * 128, sw128_desc(qa + off), sw128_desc(ka + off), idesc,
                   kk > 0 ? 1u : 0u);
        }
        mma_commit(s_full + x);
      };
      auto issue_pv = [&](int x, int j) {
        const uint32_t va = smem_u32(sKV + (j % AT_STAGES) * 2 * AT_TILE + AT_TILE);
#pragma unroll
        for (int kk = 0; kk < AT_N / 16; ++kk) {
          const uint32_t off = (kk >> 2) * AT_CHUNK + (kk & 3) * 32;
          mma_bf16_ts(tmem + 256 + x * 128, tmem + x * 128 + kk * 8, sw128_desc(va + off), idesc,
                      (j > 0 || kk > 0) ? 1u : 0u);
        }
      };
      bool ok = mbar_wait(q_full, 0, abort_flag) && mbar_wait(kv_full, 0, abort_flag);
      if (ok) {
        tc_fence_after();
        issue_s(0, 0);
        issue_s(1, 0);
      }
      for (int j = 0; j < nkb && ok; ++j) {
        const bool more = j + 1 < nkb;
        // tile A: PV_j, then S_{j+1} into the columns P_j came from (in issue order)
        if (!mbar_wait(p_full + 0, j & 1, abort_flag)) {
          ok = false;
          break;
        }
        tc_fence_after();
        issue_pv(0, j);
        if (more) {
          if (!mbar_wait(kv_full + (j + 1) % AT_STAGES, ((j + 1) / AT_STAGES) & 1, abort_flag)) {
            ok = false;
            break;
          }
          tc_fence_after();
          issue_s(0, j + 1);
        } else {
          mma_commit(o_done + 0);
        }
        // tile B
        if (!mbar_wait(p_full + 1, j & 1, abort_flag)) {
          ok = false;
          break;
        }
        tc_fence_after();
        issue_pv(1, j);
        mma_commit(kv_empty + j % AT_STAGES);
        if (more)
          issue_s(1, j + 1);
        else
          mma_commit(o_done + 1);
      }
      mma_commit(drain);
      const uint64_t t0 = global_ns();
      while (!mbar_try_wait(drain, 0) && global_ns() - t0 < kWaitLimitNs) {
      }
    }
  } else {
    // ---------------- softmax warpgroups (warps 2..5: tile A, 6..9: tile B) ----------------
    const int x = (warp - 2) >> 2;
    const int quad = warp & 3;
    const int row = quad * 32 + lane;
    const uint32_t lane_base = (uint32_t)(quad * 32) << 16;
    const uint32_t s_addr = tmem + lane_base + x * 128;
    const uint32_t o_addr = tmem + lane_base + 256 + x * 128;
    float m_use = -INFINITY, l = 0.f;
    bool ok = true;
    for (int j = 0; j < nkb; ++j) {
      const bool w = mbar_wait(s_full + x, j & 1, abort_flag);
      if (!__all_sync(0xffffffffu, w)) {
        ok = false;
        break;
      }
      tc_fence_after();
      const int kvalid = p.nk - j * AT_N;  // keys of this tile that exist (< 128 only at the end)
      // the whole S row in registers: four loads, one wait
      uint32_t r[AT_N];
#pragma unroll
      for (int c = 0; c < AT_N / 32; ++c) tmem_ld32_nowait(s_addr + c * 32, r + c * 32);
      tmem_ld_wait();
      if (kvalid < AT_N) {
#pragma unroll
        for (int i = 0; i < AT_N; ++i)
          if (i >= kvalid) r[i] = __float_as_uint(-INFINITY);
      }
      // row maximum: four independent chains of three-input maxima
      float mq[4];
#pragma unroll
      for (int u = 0; u < 4; ++u) mq[u] = fmaxf(__uint_as_float(r[2 * u]), __uint_as_float(r[2 * u + 1]));
#pragma unroll
      for (int i = 8; i < AT_N; i += 8)
#pragma unroll
        for (int u = 0; u < 4; ++u)
          mq[u] = max3(mq[u], __uint_as_float(r[i + 2 * u]), __uint_as_float(r[i + 2 * u + 1]));
      const float mx = fmaxf(fmaxf(mq[0], mq[1]), fmaxf(mq[2], mq[3]));
      const float mx2 = mx * p.scale_log2;
      float alpha = 1.f;
      if (mx2 > m_use + 8.f) {
        alpha = ex2(m_use - mx2);
        m_use = mx2;
        l *= alpha;
      }
      // P = exp2(s * scale - m) (masked keys give exp2(-inf) = 0), packed 16-bit pairs
      // written over the S columns already read
      float ls0 = 0.f, ls1 = 0.f;
#pragma unroll
      for (int c = 0; c < AT_N / 32; ++c) {
        uint32_t pk[16];
#pragma unroll
        for (int i = 0; i < 32; i += 2) {
          float x0, x1;
          fma2(x0, x1, __uint_as_float(r[c * 32 + i]), __uint_as_float(r[c * 32 + i + 1]),
               p.scale_log2, -m_use);
          const float a0 = ex2(x0), a1 = ex2(x1);
          add2(ls0, ls1, a0, a1);
          pk[i / 2] = F16 ? pack_f16x2(a0, a1) : pack_bf16x2(a0, a1);
        }
        tmem_st16(s_addr + c * 16, pk);
      }
      l += ls0 + ls1;
      // O_x holds PV of every earlier key tile (the S of this tile was issued after it);
      // rescale it before this tile's PV is issued
      if (j > 0 && __any_sync(0xffffffffu, alpha != 1.f)) {
#pragma unroll 1
        for (int c = 0; c < AT_D / 32; ++c) {
          float o[32];
          tmem_ld32(o_addr + c * 32, o);
#pragma unroll
          for (int i = 0; i < 32; ++i) o[i] *= alpha;
          tmem_st32(o_addr + c * 32, o);
        }
      }
      tmem_st_wait();
      tc_fence_before();
      mbar_arrive(p_full + x);
    }
    if (ok) {
      const bool w = mbar_wait(o_done + x, 0, abort_flag);
      if (__all_sync(0xffffffffu, w)) {
        tc_fence_after();
        const float inv = 1.f / l;
        const int q = q0 + x * AT_M + row;
        void* o1 = br ? p.o_b1 : p.o;
        void* o2 = br ? p.o2_b1 : p.o2;
        void* ob = (o2 && q >= p.o_split) ? o2 : o1;
        __nv_bfloat16* orow = reinterpret_cast<__nv_bfloat16*>(ob) + (long)q * p.ldo + head * AT_D;
#pragma unroll 1
        for (int c = 0; c < AT_D / 32; ++c) {
          float o[32];
          tmem_ld32(o_addr + c * 32, o);
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
  cudaError_t r = cudaFuncSetAttribute(attn_tc_kernel<false>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       AT_SMEM);
  if (r == cudaSuccess)
    r = cudaFuncSetAttribute(attn_tc_kernel<true>, cudaFuncAttributeMaxDynamicSharedMemorySize, AT_SMEM);
  return r;
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
  const int nbr = a.nbr > 1 ? 2 : 1;
  // with two branches the maps span both (the rows past a branch's last query or key are
  // never stored, resp. masked, and its V^T block is zero beyond nk up to vpad)
  const uint64_t qrows = nbr > 1 ? (uint64_t)a.br_q_rows + a.nq : (uint64_t)a.nq;
  const uint64_t krows = nbr > 1 ? (uint64_t)a.br_k_rows + a.nk : (uint64_t)a.nk;
  if (encode_tmap_2d_bf16(&tq, a.q, width, qrows, (uint64_t)a.ldq * 2, 64, AT_M) ||
      encode_tmap_2d_bf16(&tk, a.k, width, krows, (uint64_t)a.ldk * 2, 64, AT_N) ||
      encode_tmap_2d_bf16(&tv, a.v, (uint64_t)a.nk, width * nbr, (uint64_t)a.vpad * 2, 64, AT_D))
    return cudaErrorInvalidValue;
  AttnTcParams p;
  p.nq = a.nq;
  p.nk = a.nk;
  p.o = a.o;
  p.ldo = a.ldo;
  p.o2 = a.o2;
  p.o_split = a.o_split;
  p.br_q_rows = nbr > 1 ? (int)a.br_q_rows : 0;
  p.br_k_rows = nbr > 1 ? (int)a.br_k_rows : 0;
  p.br_v_rows = nbr > 1 ? (int)width : 0;
  p.o_b1 = a.o_b1;
  p.o2_b1 = a.o2_b1;
  p.scale_log2 = (float)(1.4426950408889634 / std::sqrt((double)AT_D));
  p.st = a.st;
  p.flag_want = a.flag_want;
  p.err = err;
  dim3 grid((a.nq + 2 * AT_M - 1) / (2 * AT_M), a.heads, nbr);
  if (a.f16)
    launch_kernel(attn_tc_kernel<true>, grid, AT_THREADS, AT_SMEM, s, tq, tk, tv, p);
  else
    launch_kernel(attn_tc_kernel<false>, grid, AT_THREADS, AT_SMEM, s, tq, tk, tv, p);
  return cudaGetLastError();
}

}  // namespace bag
