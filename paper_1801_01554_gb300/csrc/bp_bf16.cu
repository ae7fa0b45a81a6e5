// bfloat16 back-propagation step on the sm_103a tensor cores.
//
// Every contraction of the step is a GEMM C[M,N] = A[M,K] * B[N,K]^T with both
// operands K-major in global memory, fed by TMA (128-byte swizzle) into a
// multi-stage shared-memory ring, multiplied by tcgen05.mma (kind::f16, bf16
// in, fp32 accumulate) into a double-buffered TMEM accumulator, and finished
// by an epilogue that reads TMEM with tcgen05.ld:
//
//   forward  (Section 3)      A_l  = sigma(A_{l-1} W_l^T + b_l)
//                               epilogue: bias, logistic, bf16 stores of A_l
//                               row-major and transposed
//   output   (Sections 3, 8)  o = sigma(...); delta_L = (t - o) o (1 - o);
//                               error sum; bias-gradient column sums
//   hidden delta (Section 3)  delta_{l-1} = (delta_l W_l) * a (1 - a), for
//                               l = L..2 only: no delta for the input units
//                               (Section 6.1)
//   pooled change (Sec. 4.1)  G_l = delta_l^T A_{l-1}, K = the batch, split
//                               over K into fp32 partial sums
//
// The transposed copies (A_l^T, delta_l^T, X^T, W_l^T) keep every operand
// K-major.  The update kernel sums the partial changes, applies the momentum
// rule of Section 6.2.1 to the fp32 master weights and rewrites both bf16
// weight copies.  All device-side waits are bounded and latch kFlagTimeout.
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <cudaTypedefs.h>

#include <cmath>
#include <cstdio>
#include <cstring>
#include <mutex>
#include <string>
#include <vector>

#include "bp_bf16.h"
#include "bp_internal.h"

namespace bp {
namespace {

using bf16 = __nv_bfloat16;

constexpr int BM = 128;   // rows of a tile (TMEM lanes)
constexpr int BK = 64;    // K per stage: 64 bf16 = one 128-byte swizzle row
constexpr int UMMA_K = 16;
constexpr int kEpiWarps = 8;         // two per TMEM lane quarter, each on half of the columns
constexpr int kEpiThreads = 32 * kEpiWarps;
constexpr int kGemmThreads = 64 + kEpiThreads;   // warp 0 TMA, warp 1 MMA, warps 2.. epilogue

constexpr unsigned long long kWaitNs = 2000000000ull;
constexpr unsigned kWaitIters = 1u << 28;

enum Mode : int { MODE_FWD = 0, MODE_FWD_OUT = 1, MODE_DX = 2, MODE_DW = 3 };

struct GemmArgs {
    int M, N, K;
    int num_m, num_n;       // tiles along M and N
    int splits;             // K splits (pooled change only)
    int kb_per_split;       // K blocks per split
    int kb_total;
    const float* bias;      // [N]                          FWD, FWD_OUT
    bf16* out;              // [M, ldo] row-major            FWD: A_l; FWD_OUT: A_L; DX: delta
    int ldo;
    bf16* out2;             // [M, ld2] row-major            FWD_OUT: delta_L
    int ld2;
    bf16* out_t;            // [N, ldt] transposed           FWD: A_l^T; FWD_OUT/DX: delta^T
    int ldt;
    const bf16* aux;        // FWD_OUT: T [M, ld_aux]; DX: A_{l-1} [M, ld_aux]
    int ld_aux;
    float* gpart;           // DW: [splits, M, N]
    float* bias_part;       // [num_m, N]                    FWD_OUT (with T), DX
    float* sse_part;        // [num_m * num_n]               FWD_OUT (with T)
    int* flags;
};

// ------------------------------------------------------------ PTX helpers
__device__ __forceinline__ uint32_t smem_u32(const void* p) {
    return (uint32_t)__cvta_generic_to_shared(p);
}
__device__ __forceinline__ unsigned long long global_ns() {
    unsigned long long t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}
__device__ __forceinline__ void mbar_init(uint64_t* bar, unsigned count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count)
                 : "memory");
}
__device__ __forceinline__ void mbar_expect_tx(uint64_t* bar, unsigned bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)),
                 "r"(bytes)
                 : "memory");
}
__device__ __forceinline__ void mbar_arrive(uint64_t* bar) {
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}
__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, unsigned parity) {
    unsigned done;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(done)
        : "r"(smem_u32(bar)), "r"(parity)
        : "memory");
    return done != 0;
}
// Bounded wait.  Returns false if it ran out or another role aborted.
__device__ __forceinline__ bool mbar_wait(uint64_t* bar, unsigned parity, volatile int* abort_flag,
                                          int* flags) {
    if (mbar_try_wait(bar, parity)) return true;
    const unsigned long long t0 = global_ns();
    for (unsigned it = 1; it < kWaitIters; ++it) {
        if (mbar_try_wait(bar, parity)) return true;
        if ((it & 255u) == 0) {
            if (*abort_flag) return false;
            if (global_ns() - t0 > kWaitNs) break;
        }
    }
    *abort_flag = 1;
    atomicOr(flags, kFlagTimeout);
    return false;
}

__device__ __forceinline__ void tma_load_2d(void* smem_dst, const CUtensorMap* map, int c0, int c1,
                                            uint64_t* bar) {
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes "
        "[%0], [%1, {%2, %3}], [%4];" ::"r"(smem_u32(smem_dst)),
        "l"((unsigned long long)map), "r"(c0), "r"(c1), "r"(smem_u32(bar))
        : "memory");
}

// Shared-memory matrix descriptor: K-major operand, 128-byte swizzle, rows of
// 128 bytes, 8-row groups 1024 bytes apart (tcgen05 descriptor version 1).
__device__ __forceinline__ uint64_t smem_desc_sw128(uint32_t addr) {
    uint64_t d = 0;
    d |= (uint64_t)((addr & 0x3FFFFu) >> 4);
    d |= (uint64_t)(16u >> 4) << 16;      // leading byte offset (unused for this layout)
    d |= (uint64_t)(1024u >> 4) << 32;    // stride byte offset: next 8-row group
    d |= (uint64_t)1 << 46;               // descriptor version
    d |= (uint64_t)2 << 61;               // 128-byte swizzle
    return d;
}

// Instruction descriptor of tcgen05.mma kind::f16: bf16 A and B, fp32 D,
// both operands K-major, M x N tile.
__host__ __device__ constexpr uint32_t idesc_bf16(int M, int N) {
    return (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(N >> 3) << 17) |
           ((uint32_t)(M >> 4) << 24);
}

__device__ __forceinline__ void umma_bf16(uint32_t tmem_d, uint64_t adesc, uint64_t bdesc,
                                          uint32_t idesc, uint32_t accumulate) {
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "setp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(tmem_d),
        "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
        : "memory");
}
__device__ __forceinline__ void umma_commit(uint64_t* bar) {
    asm volatile(
        "tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
            smem_u32(bar))
        : "memory");
}
__device__ __forceinline__ void tc_fence_before() {
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_after() {
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}

// 32 lanes x 32 consecutive fp32 columns from TMEM.
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, float (&v)[32]) {
    uint32_t r[32];
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
        "{%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, "
        "%16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31}, [%32];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
          "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]),
          "=r"(r[14]), "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]),
          "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]), "=r"(r[25]),
          "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
        : "r"(taddr));
    asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
    for (int i = 0; i < 32; ++i) v[i] = __uint_as_float(r[i]);
}

// Logistic for bf16 outputs: hardware exp2 and the fast reciprocal divide (2 ulp;
// an IEEE divide here cost a quarter of a training step in the epilogues).
// For 1 + e^-x beyond 2^126 the quotient is 0, the logistic's value there.
__device__ __forceinline__ float sigmoid_fast(float x) { return __fdividef(1.0f, 1.0f + __expf(-x)); }

__device__ __forceinline__ float bf16_round(float x) {
    return __bfloat162float(__float2bfloat16_rn(x));
}

// Afterwards lane k holds in v[0] the warp sum of value k (31 shuffles).
__device__ __forceinline__ void reduce_scatter32(float (&v)[32], int lane) {
#pragma unroll
    for (int half = 16; half >= 1; half >>= 1) {
        const bool up = (lane & half) != 0;
#pragma unroll
        for (int k = 0; k < half; ++k) {
            const float send = up ? v[k] : v[k + half];
            const float keep = up ? v[k + half] : v[k];
            v[k] = keep + __shfl_xor_sync(0xffffffffu, send, half);
        }
    }
}

__device__ __forceinline__ void epi_bar() { asm volatile("bar.sync 1, %0;" ::"n"(kEpiThreads) : "memory"); }

// ------------------------------------------------------------ epilogue
// 32 consecutive bf16 of one row as floats (16-byte loads when the row segment is whole).
__device__ __forceinline__ void load_row32(float (&a)[32], const bf16* p, bool whole, int valid) {
    if (whole) {
#pragma unroll
        for (int k = 0; k < 4; ++k) {
            const uint4 u = __ldg(reinterpret_cast<const uint4*>(p) + k);
            const __nv_bfloat162* h = reinterpret_cast<const __nv_bfloat162*>(&u);
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                const float2 f = __bfloat1622float2(h[q]);
                a[k * 8 + 2 * q] = f.x;
                a[k * 8 + 2 * q + 1] = f.y;
            }
        }
    } else {
#pragma unroll
        for (int c = 0; c < 32; ++c) a[c] = (c < valid) ? __bfloat162float(p[c]) : 0.f;
    }
}

// One 32-column chunk of the tile for the 32 rows of one epilogue warp (this
// lane's row m).  Values are rounded to bf16 and staged in the warp's 2 KB
// shared-memory block, first by rows (16-byte pieces permuted by row so that
// the lanes' writes hit distinct banks), then transposed.  After each staging
// the warp writes every 64-byte row (or column) segment with four lanes'
// 16-byte stores, eight segments per instruction.  The column sums of a delta
// block (bias change) are read back from the transposed block.
template <int MODE>
__device__ __forceinline__ void epilogue_chunk(const GemmArgs& g, int m, int m0, int n0, int split,
                                               float (&v)[32], float& sse, bool row_ok, bf16* sS,
                                               const float* sbias, float* colsum_slot) {
    const int N = g.N;
    const int lane = threadIdx.x & 31;
    if (MODE == MODE_DW) {
        if (row_ok) {
            float* dst = g.gpart + ((size_t)split * g.M + m) * N + n0;
            if (n0 + 32 <= N && (N & 3) == 0) {
#pragma unroll
                for (int c = 0; c < 32; c += 4)
                    *reinterpret_cast<float4*>(dst + c) = make_float4(v[c], v[c + 1], v[c + 2], v[c + 3]);
            } else {
                for (int c = 0; c < 32; ++c)
                    if (n0 + c < N) dst[c] = v[c];
            }
        }
        return;
    }
    const bool whole = (n0 + 32 <= N);
    const int valid = min(32, N - n0);
    const bool with_t = (MODE == MODE_FWD_OUT) && (g.aux != nullptr);
    float vals[32];
    if (MODE == MODE_FWD || MODE == MODE_FWD_OUT) {
        float b[32];   // the tile's biases, staged in shared memory (0 past N)
#pragma unroll
        for (int k = 0; k < 8; ++k) {
            const float4 f = reinterpret_cast<const float4*>(sbias)[k];
            b[4 * k] = f.x;
            b[4 * k + 1] = f.y;
            b[4 * k + 2] = f.z;
            b[4 * k + 3] = f.w;
        }
        float t[32];
        if (with_t) load_row32(t, g.aux + (size_t)m * g.ld_aux + n0, whole && row_ok, row_ok ? valid : 0);
#pragma unroll
        for (int c = 0; c < 32; ++c) {
            const bool ok = row_ok && (c < valid);
            const float o = bf16_round(sigmoid_fast(v[c] + b[c]));
            if (with_t) {
                const float err = t[c] - o;
                sse = ok ? fmaf(err, err, sse) : sse;
                vals[c] = ok ? bf16_round(err * o * (1.f - o)) : 0.f;
            } else {
                vals[c] = ok ? o : 0.f;
            }
        }
    } else {   // MODE_DX: delta_{l-1} = (delta_l W_l) a (1 - a)
        float a[32];
        load_row32(a, g.aux + (size_t)m * g.ld_aux + n0, whole && row_ok, row_ok ? valid : 0);
#pragma unroll
        for (int c = 0; c < 32; ++c) {
            const bool ok = row_ok && (c < valid);
            vals[c] = ok ? bf16_round(v[c] * a[c] * (1.f - a[c])) : 0.f;
        }
    }
    // rows: A_l, A_L or delta_L (training output layer), or delta_{l-1}
    bf16* const rows = with_t ? g.out2 : g.out;
    const int ldr = with_t ? g.ld2 : g.ldo;
    const bool has_r = rows != nullptr;
    const bool has_t = (MODE == MODE_FWD && g.out_t != nullptr) || with_t || (MODE == MODE_DX);
    uint4* sS4 = reinterpret_cast<uint4*>(sS);
    const int piece = lane & 3;   // 16-byte piece of a 64-byte segment
    if (has_r) {
#pragma unroll
        for (int k = 0; k < 4; ++k) {
            __align__(16) __nv_bfloat162 h[4];
#pragma unroll
            for (int q = 0; q < 4; ++q) h[q] = __floats2bfloat162_rn(vals[8 * k + 2 * q], vals[8 * k + 2 * q + 1]);
            sS4[lane * 4 + (k ^ ((lane >> 1) & 3))] = *reinterpret_cast<const uint4*>(h);
        }
        __syncwarp();
        const int pieces = valid >> 3;   // N is a multiple of 8
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            const int r = j * 8 + (lane >> 2);
            if (m0 + r < g.M && piece < pieces)
                *reinterpret_cast<uint4*>(rows + (size_t)(m0 + r) * ldr + n0 + piece * 8) =
                    sS4[r * 4 + (piece ^ ((r >> 1) & 3))];
        }
        __syncwarp();   // the block is rewritten below
    }
    if (has_t) {
#pragma unroll
        for (int c = 0; c < 32; ++c) sS[c * 32 + lane] = __float2bfloat16_rn(vals[c]);
        __syncwarp();
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            const int c = j * 8 + (lane >> 2);
            const int left = g.M - (m0 + piece * 8);   // rows of this piece inside the batch
            if (c < valid && left > 0) {
                const uint4 u = sS4[c * 4 + piece];
                bf16* dst = g.out_t + (size_t)(n0 + c) * g.ldt + m0 + piece * 8;
                if (left >= 8) {
                    *reinterpret_cast<uint4*>(dst) = u;
                } else {
                    const bf16* e = reinterpret_cast<const bf16*>(&u);
#pragma unroll
                    for (int i = 0; i < 8; ++i)
                        if (i < left) dst[i] = e[i];
                }
            }
        }
    }
    if (colsum_slot != nullptr) {
        // lane c sums column c of the block over the warp's 32 rows
        const uint4* col = reinterpret_cast<const uint4*>(sS + lane * 32);
        float sum = 0.f;
#pragma unroll
        for (int k = 0; k < 4; ++k) {
            const uint4 u = col[k];
            const __nv_bfloat162* h = reinterpret_cast<const __nv_bfloat162*>(&u);
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                const float2 f = __bfloat1622float2(h[q]);
                sum += f.x;
                sum += f.y;
            }
        }
        colsum_slot[lane] = sum;
    }
    __syncwarp();   // the staging blocks may be rewritten
}

// ------------------------------------------------------------ GEMM kernel
// Tile order: groups of kGroupM row blocks, each group swept over all column
// blocks (row block fastest), so that the tiles in flight on the 152 SMs share
// a few row blocks of A and column blocks of B, which stay in L2, instead of
// reading every row block of A at once (4, 8, 16 and 32 row blocks measured
// within 2% of each other; one row block at a time was 10% slower for 4096^5).
constexpr int kGroupM = 4;
__device__ __forceinline__ void tile_coords(int tile, int num_m, int num_n, int& mb, int& nb) {
    const int per_group = kGroupM * num_n;
    const int grp = tile / per_group;
    const int first = grp * kGroupM;
    const int gm = min(num_m - first, kGroupM);
    const int local = tile - grp * per_group;
    mb = first + local % gm;
    nb = local / gm;
}

template <int BN, int MODE>
struct GemmCfg {
    static constexpr int kStages = BN == 256 ? 4 : 6;
    static constexpr int kABytes = BM * BK * 2;
    static constexpr int kBBytes = BN * BK * 2;
    static constexpr int kStageBytes = kABytes + kBBytes;
    static constexpr int kTmemCols = 2 * BN;   // two accumulators
    // tile ring, then barriers and scratch
    static constexpr int kRingBytes = kStages * kStageBytes;
    static constexpr int kColsumBytes = 4 * BN * 4;
    static constexpr int kStageOutBytes = kEpiWarps * 32 * 32 * 2;   // one 32 x 32 bf16 block per epilogue warp
    static constexpr int kBiasBytes = 2 * BN * 4;   // the tile's biases, one block per accumulator
    static constexpr int kSmemBytes =
        1024 + kRingBytes + kColsumBytes + kStageOutBytes + kBiasBytes + 256;
};

template <int BN, int MODE>
__global__ void __launch_bounds__(kGemmThreads, 1)
    k_gemm(const __grid_constant__ CUtensorMap map_a, const __grid_constant__ CUtensorMap map_b,
           GemmArgs g) {
    using Cfg = GemmCfg<BN, MODE>;
    constexpr int S = Cfg::kStages;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
    uint8_t* ring = smem;
    float* colsum = reinterpret_cast<float*>(smem + Cfg::kRingBytes);   // [4][BN]
    bf16* stage_out = reinterpret_cast<bf16*>(smem + Cfg::kRingBytes + Cfg::kColsumBytes);
    float* bias_s = reinterpret_cast<float*>(smem + Cfg::kRingBytes + Cfg::kColsumBytes +
                                             Cfg::kStageOutBytes);   // [2][BN]
    uint64_t* bars = reinterpret_cast<uint64_t*>(smem + Cfg::kRingBytes + Cfg::kColsumBytes +
                                                 Cfg::kStageOutBytes + Cfg::kBiasBytes);
    uint64_t* full = bars;              // [S]
    uint64_t* empty = bars + S;         // [S]
    uint64_t* tfull = bars + 2 * S;     // [2]
    uint64_t* tempty = bars + 2 * S + 2;   // [2]
    uint64_t* drain = bars + 2 * S + 4;    // [1] used only when a wait ran out
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 2 * S + 5);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int tiles = g.num_m * g.num_n;
    const int items = tiles * g.splits;

    if (threadIdx.x == 0) {
        for (int s = 0; s < S; ++s) {
            mbar_init(&full[s], 1);
            mbar_init(&empty[s], 1);
        }
        for (int a = 0; a < 2; ++a) {
            mbar_init(&tfull[a], 1);
            mbar_init(&tempty[a], kEpiThreads);
        }
        mbar_init(drain, 1);
        *abort_flag = 0;
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    if (warp == 1) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                         smem_u32(tmem_slot)),
                     "r"(Cfg::kTmemCols)
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem_base = *tmem_slot;

    if (warp == 0) {
        // ---------------- TMA producer
        if (lane == 0) {
            int stage = 0;
            unsigned phase = 0;
            int issued_parity[8];
            for (int s = 0; s < S; ++s) issued_parity[s] = -1;
            bool ok = true;
            for (int it = blockIdx.x; it < items && ok; it += gridDim.x) {
                const int tile = it % tiles, split = it / tiles;
                int mb, nb;
                tile_coords(tile, g.num_m, g.num_n, mb, nb);
                const int kb0 = split * g.kb_per_split;
                const int kb1 = min(g.kb_total, kb0 + g.kb_per_split);
                for (int kb = kb0; kb < kb1; ++kb) {
                    if (!mbar_wait(&empty[stage], phase ^ 1u, abort_flag, g.flags)) { ok = false; break; }
                    uint8_t* sa = ring + stage * Cfg::kStageBytes;
                    uint8_t* sb = sa + Cfg::kABytes;
                    mbar_expect_tx(&full[stage], Cfg::kStageBytes);
                    tma_load_2d(sa, &map_a, kb * BK, mb * BM, &full[stage]);
                    tma_load_2d(sb, &map_b, kb * BK, nb * BN, &full[stage]);
                    issued_parity[stage] = (int)phase;
                    if (++stage == S) { stage = 0; phase ^= 1u; }
                }
            }
            if (!ok) {
                // let every copy already issued land before the CTA can exit
                for (int s = 0; s < S; ++s) {
                    if (issued_parity[s] < 0) continue;
                    const unsigned long long t0 = global_ns();
                    while (!mbar_try_wait(&full[s], (unsigned)issued_parity[s]) &&
                           global_ns() - t0 < kWaitNs) {
                    }
                }
            }
        }
    } else if (warp == 1) {
        // ---------------- MMA issuer
        if (lane == 0) {
            constexpr uint32_t idesc = idesc_bf16(BM, BN);
            int stage = 0;
            unsigned phase = 0;
            int acc = 0;
            unsigned acc_phase = 0;
            bool ok = true;
            bool issued_any = false;
            for (int it = blockIdx.x; it < items && ok; it += gridDim.x) {
                const int split = it / tiles;
                const int kb0 = split * g.kb_per_split;
                const int kb1 = min(g.kb_total, kb0 + g.kb_per_split);
                if (!mbar_wait(&tempty[acc], acc_phase ^ 1u, abort_flag, g.flags)) { ok = false; break; }
                tc_fence_after();
                const uint32_t tmem_d = tmem_base + (uint32_t)(acc * BN);
                for (int kb = kb0; kb < kb1; ++kb) {
                    if (!mbar_wait(&full[stage], phase, abort_flag, g.flags)) { ok = false; break; }
                    tc_fence_after();
                    const uint32_t a0 = smem_u32(ring + stage * Cfg::kStageBytes);
                    const uint32_t b0 = a0 + Cfg::kABytes;
#pragma unroll
                    for (int kk = 0; kk < BK / UMMA_K; ++kk) {
                        const uint64_t ad = smem_desc_sw128(a0 + kk * UMMA_K * 2);
                        const uint64_t bd = smem_desc_sw128(b0 + kk * UMMA_K * 2);
                        umma_bf16(tmem_d, ad, bd, idesc, (kb > kb0 || kk > 0) ? 1u : 0u);
                    }
                    issued_any = true;
                    umma_commit(&empty[stage]);
                    if (++stage == S) { stage = 0; phase ^= 1u; }
                }
                if (!ok) break;
                umma_commit(&tfull[acc]);
                if (++acc == 2) { acc = 0; acc_phase ^= 1u; }
            }
            if (!ok && issued_any) {
                // let every MMA already issued finish before TMEM is released
                umma_commit(drain);
                const unsigned long long t0 = global_ns();
                while (!mbar_try_wait(drain, 0) && global_ns() - t0 < kWaitNs) {
                }
            }
        }
    } else {
        // ---------------- epilogue warps 2..9
        const int q = warp & 3;                  // TMEM lane quarter this warp may access
        const int ew = warp - 2;                 // 0..7
        const int slot = ew & 3;                 // row quarter's slot in the column-sum scratch
        const int cbeg = (ew >> 2) * (BN / 2);   // this warp's half of the columns
        int acc = 0;
        unsigned acc_phase = 0;
        for (int it = blockIdx.x; it < items; it += gridDim.x) {
            const int tile = it % tiles, split = it / tiles;
            int mb, nb;
            tile_coords(tile, g.num_m, g.num_n, mb, nb);
            float* sbias = bias_s + acc * BN;
            if (MODE == MODE_FWD || MODE == MODE_FWD_OUT) {
                // block acc was last read two tiles ago, before the barrier of the previous tile
                for (int c = threadIdx.x - 64; c < BN; c += kEpiThreads) {
                    const int n = nb * BN + c;
                    sbias[c] = n < g.N ? __ldg(g.bias + n) : 0.f;
                }
            }
            mbar_wait(&tfull[acc], acc_phase, abort_flag, g.flags);
            epi_bar();                     // the epilogue warps leave together on an abort
            if (*abort_flag) break;
            tc_fence_after();
            const int m = mb * BM + q * 32 + lane;
            const bool row_ok = m < g.M;
            float sse = 0.f;
            const uint32_t tbase = tmem_base + ((uint32_t)(q * 32) << 16) + (uint32_t)(acc * BN);
            const int m0 = mb * BM + q * 32;
            bf16* sS = stage_out + ew * 1024;
            const bool want_colsum = (MODE == MODE_DX) || (MODE == MODE_FWD_OUT && g.aux != nullptr);
            for (int c0 = cbeg; c0 < cbeg + BN / 2; c0 += 32) {
                const int n0 = nb * BN + c0;
                float v[32];
                tmem_ld32(tbase + (uint32_t)c0, v);
                if (n0 >= g.N) {
                    if (want_colsum) colsum[slot * BN + c0 + lane] = 0.f;
                    continue;
                }
                epilogue_chunk<MODE>(g, m, m0, n0, split, v, sse, row_ok, sS, sbias + c0,
                                     want_colsum ? colsum + slot * BN + c0 : nullptr);
            }
            // TMEM is free for the next accumulation into this buffer
            tc_fence_before();
            mbar_arrive(&tempty[acc]);
            if (++acc == 2) { acc = 0; acc_phase ^= 1u; }
            if (MODE == MODE_DX || (MODE == MODE_FWD_OUT && g.aux != nullptr)) {
                epi_bar();
                const int t = threadIdx.x - 64;   // 0 .. kEpiThreads - 1
                for (int c = t; c < BN; c += kEpiThreads) {
                    const int n = nb * BN + c;
                    if (n < g.N) {
                        const float s = (colsum[c] + colsum[BN + c]) + (colsum[2 * BN + c] + colsum[3 * BN + c]);
                        g.bias_part[(size_t)mb * g.N + n] = s;
                    }
                }
                if (MODE == MODE_FWD_OUT) {
                    // tile error sum: warp sums, then the eight warps in a fixed order
#pragma unroll
                    for (int o = 16; o > 0; o >>= 1) sse += __shfl_xor_sync(0xffffffffu, sse, o);
                    epi_bar();
                    if (lane == 0) colsum[ew] = sse;
                    epi_bar();
                    if (t == 0)
                        g.sse_part[tile] = ((colsum[0] + colsum[1]) + (colsum[2] + colsum[3])) +
                                           ((colsum[4] + colsum[5]) + (colsum[6] + colsum[7]));
                }
                epi_bar();
            }
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem_base),
                     "r"(Cfg::kTmemCols)
                     : "memory");
    }
}

// ------------------------------------------------------------ SIMT kernels
// dst[c][r] = src[r][c] for a [rows, cols] bf16 matrix whose column count and
// both pitches are multiples of 8 (64 x 64 tiles, 256 threads).  Rows of src
// and of dst move in 16-byte pieces; the shared-memory pitch of 33 words keeps
// the lanes' 4-byte writes conflict-free.
__global__ void __launch_bounds__(256) k_transpose(const bf16* __restrict__ src, int rows, int cols,
                                                   int lds, bf16* __restrict__ dst, int ldd) {
    __shared__ __align__(16) uint32_t tile[64][33];   // [r][pair of columns]
    const int c0 = blockIdx.x * 64, r0 = blockIdx.y * 64;
    const int t = threadIdx.x, p = t & 7;
#pragma unroll
    for (int h = 0; h < 2; ++h) {
        const int r = (t >> 3) + 32 * h, c = c0 + p * 8;
        uint4 u = make_uint4(0u, 0u, 0u, 0u);
        if (r0 + r < rows && c < cols) u = *reinterpret_cast<const uint4*>(src + (size_t)(r0 + r) * lds + c);
        tile[r][p * 4] = u.x;
        tile[r][p * 4 + 1] = u.y;
        tile[r][p * 4 + 2] = u.z;
        tile[r][p * 4 + 3] = u.w;
    }
    __syncthreads();
    const bf16* tb = reinterpret_cast<const bf16*>(&tile[0][0]);   // element (r, c) at r * 66 + c
#pragma unroll
    for (int h = 0; h < 2; ++h) {
        const int c = (t >> 3) + 32 * h, r = p * 8;   // dst row c0 + c, columns r0 + r .. +7
        if (c0 + c >= cols || r0 + r >= rows) continue;
        __align__(16) bf16 e[8];
#pragma unroll
        for (int k = 0; k < 8; ++k) e[k] = tb[(r + k) * 66 + c];
        bf16* d = dst + (size_t)(c0 + c) * ldd + r0 + r;
        if (r0 + r + 8 <= rows) {
            *reinterpret_cast<uint4*>(d) = *reinterpret_cast<const uint4*>(e);
        } else {
#pragma unroll
            for (int k = 0; k < 8; ++k)
                if (r0 + r + k < rows) d[k] = e[k];
        }
    }
}

// Output deltas from stored outputs (bp_backward): delta = (t - o) o (1 - o),
// delta rows and transposed copy, per-128-row column sums and error sums.
// One block of 128 threads per (128-row tile, 32-column chunk).
__global__ void k_output_delta(const bf16* __restrict__ O, const bf16* __restrict__ T, int M, int N,
                               int ld, bf16* __restrict__ Drow, bf16* __restrict__ Dt, int ldt,
                               float* __restrict__ bias_part, float* __restrict__ sse_part,
                               int num_n_chunks) {
    __shared__ float cs[4][32];
    __shared__ float ss[4];
    const int mb = blockIdx.y, nc = blockIdx.x;
    const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int m = mb * 128 + threadIdx.x;
    const bool row_ok = m < M;
    float d[32];
    float sse = 0.f;
    for (int c = 0; c < 32; ++c) {
        const int n = nc * 32 + c;
        const bool ok = row_ok && n < N;
        float dv = 0.f;
        if (ok) {
            const float o = __bfloat162float(O[(size_t)m * ld + n]);
            const float err = __bfloat162float(T[(size_t)m * ld + n]) - o;
            sse = fmaf(err, err, sse);
            dv = bf16_round(err * o * (1.f - o));
            Drow[(size_t)m * ld + n] = __float2bfloat16_rn(dv);
            Dt[(size_t)n * ldt + m] = __float2bfloat16_rn(dv);
        }
        d[c] = dv;
    }
    reduce_scatter32(d, lane);
    cs[w][lane] = d[0];
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) sse += __shfl_xor_sync(0xffffffffu, sse, o);
    if (lane == 0) ss[w] = sse;
    __syncthreads();
    if (threadIdx.x < 32) {
        const int n = nc * 32 + threadIdx.x;
        if (n < N) bias_part[(size_t)mb * N + n] = (cs[0][threadIdx.x] + cs[1][threadIdx.x]) +
                                                   (cs[2][threadIdx.x] + cs[3][threadIdx.x]);
    }
    if (threadIdx.x == 0) sse_part[(size_t)mb * num_n_chunks + nc] = (ss[0] + ss[1]) + (ss[2] + ss[3]);
}

constexpr int kUT = 64;   // update kernel: weight tile edge

struct LayerUpd {
    int n_out, n_in;
    long long woff, boff;       // offsets in theta / V / G
    const float* gpart;         // [splits, n_out, n_in] (null: none)
    int splits;
    const float* bias_part;     // [mtiles, n_out]
    int mtiles;
    bf16* wb;                   // [n_out, n_in]
    bf16* wt;                   // [n_in, n_out]
};
struct UpdArgs {
    int L;
    LayerUpd ly[kMaxL];
    int tile0[kMaxL + 1];       // kUT x kUT weight tiles (+ one bias row band) per layer
    float* theta;
    float* V;
    float* G;
    float lr_gs, momentum;
    int mode;                   // 0: apply update; 1: accumulate into G; 2: refresh bf16 copies
    int fold_g;
    const float* sse_part;
    int n_sse;
    float* sse_out;
    int* flags;
    float guard;          // > 0: fault guard of Section 8
    unsigned* faults;     // changes the guard zeroed
};

// Fault guard of Section 8: a total weight change outside (-guard, guard), or
// not a number, is set to zero and counted (off while guard <= 0).
__device__ __forceinline__ float guard_change(const UpdArgs& a, float g) {
    if (a.guard > 0.f && !(fabsf(g) <= a.guard)) {
        atomicAdd(a.faults, 1u);
        return 0.f;
    }
    return g;
}

// Momentum update of Section 6.2.1 over 64 x 64 weight tiles plus the biases:
// g = sum of partial changes (+ pending G); v = lr*gs*g + m*v; w += v; then the
// bf16 copy and its transpose.  Mode 1 adds the partial changes into G instead.
// The kernel waits on DRAM latency: three CTAs per SM (80 registers, no spill),
// and two partial planes' loads issued together, keep more bytes in flight.
__global__ void __launch_bounds__(256, 3) k_update_bf16(UpdArgs a) {
    if (blockIdx.x == 0 && threadIdx.x == 0 && a.sse_out != nullptr) {
        float s = 0.f;
        for (int k = 0; k < a.n_sse; ++k) s += a.sse_part[k];
        *a.sse_out = s;
        if (!isfinite(s)) atomicOr(a.flags, kFlagNonfinite);
    }
    const int total = a.tile0[a.L];
    for (int t = blockIdx.x; t < total; t += gridDim.x) {
        int l = 0;
        while (t >= a.tile0[l + 1]) ++l;
        const LayerUpd& u = a.ly[l];
        const int lt = t - a.tile0[l];
        const int cols = (u.n_in + kUT - 1) / kUT;
        const int rb = lt / cols, cb = lt - rb * cols;   // rb == row-tile count: the biases
        const int rows_w = (u.n_out + kUT - 1) / kUT;
        if (rb < rows_w) {
            // Warp w covers rows 16*(w/2) .. +16 and columns 32*(w%2) .. +32 of the
            // tile; a lane holds 4 consecutive rows x 4 consecutive columns, so the
            // fp32 rows move as float4 (8 lanes: one 128-byte line per row) and
            // both bf16 copies as 8-byte pieces (the transposed copy's 4 rows are
            // the lane's own).  Layer sizes are multiples of 8: a lane's 4 x 4
            // block is either inside the layer or outside it.  All loads of the
            // lane come before its stores.
            const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
            const int i = cb * kUT + (w & 1) * 32 + (lane & 7) * 4;
            const int j0 = rb * kUT + (w >> 1) * 16 + (lane >> 3) * 4;
            if (i < u.n_in && j0 < u.n_out) {
                const float4 z = make_float4(0.f, 0.f, 0.f, 0.f);
                float4 gs[4], w4[4], v4[4];
                const size_t e0 = (size_t)j0 * u.n_in + i;
                const float* th = a.theta + u.woff + e0;
                float* vv = a.V + u.woff + e0;
                float* gg = a.G + u.woff + e0;
#pragma unroll
                for (int r = 0; r < 4; ++r) {
                    gs[r] = z;
                    v4[r] = z;
                    w4[r] = *reinterpret_cast<const float4*>(th + (size_t)r * u.n_in);
                    if (a.mode == 0) v4[r] = *reinterpret_cast<const float4*>(vv + (size_t)r * u.n_in);
                }
                if (a.mode != 2) {
                    const size_t plane = (size_t)u.n_out * u.n_in;
                    int s0 = 0;
                    for (; s0 + 2 <= u.splits; s0 += 2) {
                        const float* gp = u.gpart + s0 * plane + e0;
                        float4 p0[4], p1[4];
#pragma unroll
                        for (int r = 0; r < 4; ++r) {
                            p0[r] = __ldcs(reinterpret_cast<const float4*>(gp + (size_t)r * u.n_in));
                            p1[r] = __ldcs(reinterpret_cast<const float4*>(gp + plane + (size_t)r * u.n_in));
                        }
#pragma unroll
                        for (int r = 0; r < 4; ++r) {
                            gs[r].x += p0[r].x;
                            gs[r].y += p0[r].y;
                            gs[r].z += p0[r].z;
                            gs[r].w += p0[r].w;
                            gs[r].x += p1[r].x;
                            gs[r].y += p1[r].y;
                            gs[r].z += p1[r].z;
                            gs[r].w += p1[r].w;
                        }
                    }
                    for (int s = s0; s < u.splits; ++s) {
                        const float* gp = u.gpart + s * plane + e0;
#pragma unroll
                        for (int r = 0; r < 4; ++r) {
                            const float4 p = __ldcs(reinterpret_cast<const float4*>(gp + (size_t)r * u.n_in));
                            gs[r].x += p.x;
                            gs[r].y += p.y;
                            gs[r].z += p.z;
                            gs[r].w += p.w;
                        }
                    }
                }
#pragma unroll
                for (int r = 0; r < 4; ++r) {
                    const size_t o = (size_t)r * u.n_in;
                    if (a.mode == 1) {
                        float4 g4 = *reinterpret_cast<const float4*>(gg + o);
                        g4.x += gs[r].x;
                        g4.y += gs[r].y;
                        g4.z += gs[r].z;
                        g4.w += gs[r].w;
                        *reinterpret_cast<float4*>(gg + o) = g4;
                    } else if (a.mode == 0) {
                        const float4 gp4 = a.fold_g ? *reinterpret_cast<const float4*>(gg + o) : z;
                        float* wc = &w4[r].x;
                        float* vc = &v4[r].x;
                        const float* gc = &gs[r].x;
                        const float* pc = &gp4.x;
#pragma unroll
                        for (int c = 0; c < 4; ++c) {
                            const float vel = a.lr_gs * guard_change(a, gc[c] + pc[c]) + a.momentum * vc[c];
                            vc[c] = vel;
                            wc[c] += vel;
                        }
                        *reinterpret_cast<float4*>(vv + o) = v4[r];
                        *reinterpret_cast<float4*>(a.theta + u.woff + e0 + o) = w4[r];
                        if (a.fold_g) *reinterpret_cast<float4*>(gg + o) = z;
                    }
                    if (a.mode != 1) {
                        __align__(8) __nv_bfloat162 h[2];
                        h[0] = __floats2bfloat162_rn(w4[r].x, w4[r].y);
                        h[1] = __floats2bfloat162_rn(w4[r].z, w4[r].w);
                        *reinterpret_cast<uint2*>(u.wb + e0 + o) = *reinterpret_cast<const uint2*>(h);
                    }
                }
                if (a.mode != 1) {
                    // W_l^T rows i .. i+3, columns j0 .. j0+3
#pragma unroll
                    for (int c = 0; c < 4; ++c) {
                        __align__(8) __nv_bfloat162 h[2];
                        h[0] = __floats2bfloat162_rn((&w4[0].x)[c], (&w4[1].x)[c]);
                        h[1] = __floats2bfloat162_rn((&w4[2].x)[c], (&w4[3].x)[c]);
                        *reinterpret_cast<uint2*>(u.wt + (size_t)(i + c) * u.n_out + j0) =
                            *reinterpret_cast<const uint2*>(h);
                    }
                }
            }
        } else {
            // biases of this layer, spread over the `cols` tiles of the bias row (one
            // tile with the rest idle left a long tail of dependent partial-sum loads);
            // each bias sums its row-block partials in order, loads issued 16 ahead
            const int per = (u.n_out + cols - 1) / cols;
            const int j_hi = min(u.n_out, (cb + 1) * per);
            for (int j = cb * per + threadIdx.x; j < j_hi; j += 256) {
                const long long idx = u.boff + j;
                float gsum = 0.f;
                if (a.mode != 2) {
#pragma unroll 16
                    for (int mt = 0; mt < u.mtiles; ++mt) gsum += u.bias_part[(size_t)mt * u.n_out + j];
                }
                if (a.mode == 1) {
                    a.G[idx] += gsum;
                } else if (a.mode == 0) {
                    if (a.fold_g) {
                        gsum += a.G[idx];
                        a.G[idx] = 0.f;
                    }
                    const float vel = a.lr_gs * guard_change(a, gsum) + a.momentum * a.V[idx];
                    a.V[idx] = vel;
                    a.theta[idx] += vel;
                }
            }
        }
    }
}

// ------------------------------------------------------------ host side
std::string g_msg;

PFN_cuTensorMapEncodeTiled_v12000 g_encode = nullptr;

bool get_encoder() {
    if (!g_encode) g_encode = tensor_map_encoder();
    return g_encode != nullptr;
}

// 2-D bf16 tensor map over a row-major [rows, cols] matrix with row pitch `ld`
// elements, box = box_rows x 64 columns, 128-byte swizzle, zero fill.
bool make_map(CUtensorMap* map, const void* base, int rows, int cols, int ld, int box_rows) {
    cuuint64_t dims[2] = {(cuuint64_t)cols, (cuuint64_t)rows};
    cuuint64_t strides[1] = {(cuuint64_t)ld * 2};
    cuuint32_t box[2] = {(cuuint32_t)BK, (cuuint32_t)box_rows};
    cuuint32_t estr[2] = {1, 1};
    CUresult r = g_encode(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims,
                          strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                          CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                          CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS;
}


template <int BN, int MODE>
cudaError_t gemm_setup() {
    return cudaFuncSetAttribute(k_gemm<BN, MODE>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                GemmCfg<BN, MODE>::kSmemBytes);
}

std::mutex g_mu;
bool g_ready[64];

cudaError_t setup_all(int device) {
    std::lock_guard<std::mutex> lk(g_mu);
    if (device < 64 && g_ready[device]) return cudaSuccess;
    cudaError_t e;
    if ((e = gemm_setup<256, MODE_FWD>()) != cudaSuccess) return e;
    if ((e = gemm_setup<256, MODE_FWD_OUT>()) != cudaSuccess) return e;
    if ((e = gemm_setup<256, MODE_DX>()) != cudaSuccess) return e;
    if ((e = gemm_setup<256, MODE_DW>()) != cudaSuccess) return e;
    if (device < 64) g_ready[device] = true;
    return cudaSuccess;
}

constexpr int kBN = 256;

}  // namespace

struct Bf16Net {
    int L = 0;
    int n[BP_MAX_SIZES] = {0};
    int cap = 0, cap_pad = 0;
    int num_sms = 0;
    float* theta = nullptr;
    float* V = nullptr;
    float* G = nullptr;
    int* flags = nullptr;       // [0] error bits, [1] fault-guard count
    float guard = 0.f;          // fault guard of Section 8 (0: off)
    long long woff[BP_MAX_SIZES] = {0}, boff[BP_MAX_SIZES] = {0};
    bf16* wb[BP_MAX_SIZES] = {nullptr};     // W_l   [n_l, n_{l-1}]
    bf16* wt[BP_MAX_SIZES] = {nullptr};     // W_l^T [n_{l-1}, n_l]
    bf16* act[BP_MAX_SIZES] = {nullptr};    // A_l   [cap, n_l], l >= 1
    bf16* actT[BP_MAX_SIZES] = {nullptr};   // A_l^T [n_l, cap_pad], l = 0..L-1
    bf16* dlt[BP_MAX_SIZES] = {nullptr};    // delta_l [cap, n_l], l >= 1
    bf16* dltT[BP_MAX_SIZES] = {nullptr};   // delta_l^T [n_l, cap_pad]
    float* gpart[BP_MAX_SIZES] = {nullptr}; // [splits, n_l, n_{l-1}]
    int splits[BP_MAX_SIZES] = {0};
    float* bpart[BP_MAX_SIZES] = {nullptr}; // [mtiles(cap), n_l]
    float* sse_part = nullptr;              // [mtiles(cap) * tiles along n_L]
    int n_sse_cap = 0;
    // X^T runs on a stream of the net's own, forked from and joined back into
    // the caller's stream, beside the hidden-delta GEMMs
    cudaStream_t side = nullptr;
    cudaEvent_t fork = nullptr, join = nullptr;
    std::vector<void*> allocs;
};

namespace {

bool alloc(Bf16Net* b, void** p, size_t bytes) {
    if (cudaMalloc(p, bytes) != cudaSuccess) return false;
    b->allocs.push_back(*p);
    return true;
}

int ceil_div(long long a, long long b) { return (int)((a + b - 1) / b); }

// Splits of K (the batch) for a pooled-change GEMM of `tiles` output tiles:
// the fewest that minimise, in units of one full-K tile's time on one SM,
//   ceil(tiles * s / num_sms) / s     (waves of 1/s-K work items)
//   + s * r                           (the s partial planes: written here, read by the update)
// with r = (tile bytes of fp32 partials, out and back) / (tile MMA time) =
// 8 BM BN / HBM  /  (2 BM BN K / (bf16 peak / SM)) = 4 F_sm / (K HBM); the
// measured ratio of per-SM bf16 peak to HBM bandwidth, 12.7 TFLOP/s to
// 6.8 TB/s, is 1.87 flop per byte.
int pick_splits(int tiles, int kb_total, int num_sms, int cap_splits) {
    if (tiles < 1) tiles = 1;
    const double r = 4.0 * 1.87 / ((double)kb_total * BK);
    int best = 1;
    double best_cost = 0.0;
    for (int s = 1; s <= cap_splits && s <= kb_total; ++s) {
        const double waves = (double)(((long long)tiles * s + num_sms - 1) / num_sms) / s;
        const double cost = waves + s * r * tiles;
        if (s == 1 || cost < best_cost * (1.0 - 1e-9)) {
            best = s;
            best_cost = cost;
        }
    }
    return best;
}

template <int MODE>
cudaError_t launch_gemm(const Bf16Net* b, const CUtensorMap& ma, const CUtensorMap& mb,
                        GemmArgs g, cudaStream_t s) {
    g.num_m = ceil_div(g.M, BM);
    g.num_n = ceil_div(g.N, kBN);
    g.kb_total = ceil_div(g.K, BK);
    if (g.splits < 1) g.splits = 1;
    g.kb_per_split = ceil_div(g.kb_total, g.splits);
    g.splits = ceil_div(g.kb_total, g.kb_per_split);   // every split non-empty
    g.flags = b->flags;
    const int items = g.num_m * g.num_n * g.splits;
    const int grid = items < b->num_sms ? items : b->num_sms;
    k_gemm<kBN, MODE><<<grid, kGemmThreads, GemmCfg<kBN, MODE>::kSmemBytes, s>>>(ma, mb, g);
    return cudaGetLastError();
}

GemmArgs blank_args() {
    GemmArgs g;
    memset(&g, 0, sizeof g);
    g.splits = 1;
    return g;
}

// Forward pass of all layers; with T, also the output deltas (training).
cudaError_t run_forward(Bf16Net* b, const bf16* X, int B, const bf16* T, bf16* Y, cudaStream_t s) {
    const int L = b->L;
    for (int l = 1; l <= L; ++l) {
        const bf16* A = (l == 1) ? X : b->act[l - 1];
        CUtensorMap ma, mb;
        if (!make_map(&ma, A, B, b->n[l - 1], b->n[l - 1], BM) ||
            !make_map(&mb, b->wb[l], b->n[l], b->n[l - 1], b->n[l - 1], kBN))
            return cudaErrorInvalidValue;
        GemmArgs g = blank_args();
        g.M = B;
        g.N = b->n[l];
        g.K = b->n[l - 1];
        g.bias = b->theta + b->boff[l];
        cudaError_t e;
        if (l < L) {
            g.out = b->act[l];
            g.ldo = b->n[l];
            g.out_t = b->actT[l];
            g.ldt = b->cap_pad;
            e = launch_gemm<MODE_FWD>(b, ma, mb, g, s);
        } else {
            if (T != nullptr) {
                // training: the output deltas (rows and transposed) replace the outputs
                g.aux = T;
                g.ld_aux = b->n[L];
                g.out2 = b->dlt[L];
                g.ld2 = b->n[L];
                g.out_t = b->dltT[L];
                g.ldt = b->cap_pad;
                g.bias_part = b->bpart[L];
                g.sse_part = b->sse_part;
            } else {
                g.out = (Y != nullptr) ? Y : b->act[L];
                g.ldo = b->n[L];
            }
            e = launch_gemm<MODE_FWD_OUT>(b, ma, mb, g, s);
        }
        if (e != cudaSuccess) return e;
    }
    return cudaSuccess;
}

// Hidden deltas and pooled partial changes for every layer (deltas of layer L
// and the activations must already be in scratch).
cudaError_t run_backward(Bf16Net* b, const bf16* X, int B, cudaStream_t s) {
    const int L = b->L;
    // X^T for the first layer's pooled change, on the side stream: it reads only
    // X, so it overlaps the hidden-delta GEMMs (one 8.4 KB transpose block fits
    // beside a GEMM CTA on an SM).  The fork orders it after everything already
    // on s, the previous group's read of the same buffer included; the join
    // orders the pooled-change GEMMs after it.
    {
        cudaError_t e = cudaEventRecord(b->fork, s);
        if (e == cudaSuccess) e = cudaStreamWaitEvent(b->side, b->fork, 0);
        if (e != cudaSuccess) return e;
        dim3 grid(ceil_div(b->n[0], 64), ceil_div(B, 64));
        k_transpose<<<grid, 256, 0, b->side>>>(X, B, b->n[0], b->n[0], b->actT[0], b->cap_pad);
        e = cudaGetLastError();
        if (e == cudaSuccess) e = cudaEventRecord(b->join, b->side);
        if (e != cudaSuccess) return e;
    }
    cudaError_t e_dx = cudaSuccess;
    for (int l = L; l >= 2 && e_dx == cudaSuccess; --l) {
        // delta_{l-1} = (delta_l W_l) * a (1 - a):  A = delta_l [B, n_l], B-operand = W_l^T
        CUtensorMap ma, mb;
        if (!make_map(&ma, b->dlt[l], B, b->n[l], b->n[l], BM) ||
            !make_map(&mb, b->wt[l], b->n[l - 1], b->n[l], b->n[l], kBN)) {
            e_dx = cudaErrorInvalidValue;
            break;
        }
        GemmArgs g = blank_args();
        g.M = B;
        g.N = b->n[l - 1];
        g.K = b->n[l];
        g.out = (l - 1 >= 2) ? b->dlt[l - 1] : nullptr;
        g.ldo = b->n[l - 1];
        g.out_t = b->dltT[l - 1];
        g.ldt = b->cap_pad;
        g.aux = b->act[l - 1];
        g.ld_aux = b->n[l - 1];
        g.bias_part = b->bpart[l - 1];
        e_dx = launch_gemm<MODE_DX>(b, ma, mb, g, s);
    }
    // joined on every path, so that a stream capture on s stays whole
    const cudaError_t e_join = cudaStreamWaitEvent(s, b->join, 0);
    if (e_dx != cudaSuccess) return e_dx;
    if (e_join != cudaSuccess) return e_join;
    for (int l = 1; l <= L; ++l) {
        // G_l = delta_l^T A_{l-1}: A = delta_l^T [n_l, B], B-operand = A_{l-1}^T [n_{l-1}, B]
        CUtensorMap ma, mb;
        if (!make_map(&ma, b->dltT[l], b->n[l], B, b->cap_pad, BM) ||
            !make_map(&mb, b->actT[l - 1], b->n[l - 1], B, b->cap_pad, kBN))
            return cudaErrorInvalidValue;
        GemmArgs g = blank_args();
        g.M = b->n[l];
        g.N = b->n[l - 1];
        g.K = B;
        g.gpart = b->gpart[l];
        g.splits = b->splits[l];
        const int tiles = ceil_div(g.M, BM) * ceil_div(g.N, kBN);
        g.splits = pick_splits(tiles, ceil_div(B, BK), b->num_sms, b->splits[l]);
        cudaError_t e = launch_gemm<MODE_DW>(b, ma, mb, g, s);
        if (e != cudaSuccess) return e;
    }
    return cudaSuccess;
}

// B: patterns whose partial changes are pending (0: none).
UpdArgs upd_args(Bf16Net* b, int B, int mode, bool fold, float lr_gs, float momentum, float* sse_out,
                 int n_sse) {
    UpdArgs a;
    memset(&a, 0, sizeof a);
    a.L = b->L;
    int tiles = 0;
    for (int l = 1; l <= b->L; ++l) {
        LayerUpd& u = a.ly[l - 1];
        u.n_out = b->n[l];
        u.n_in = b->n[l - 1];
        u.woff = b->woff[l];
        u.boff = b->boff[l];
        u.gpart = b->gpart[l];
        const int t = ceil_div(u.n_out, BM) * ceil_div(u.n_in, kBN);
        u.splits = 0;
        u.mtiles = 0;
        if (mode != 2 && B > 0) {
            // the same split of K = B as the pooled-change GEMM used
            const int kbt = ceil_div(B, BK);
            const int s0 = pick_splits(t, kbt, b->num_sms, b->splits[l]);
            const int kps = ceil_div(kbt, s0);
            u.splits = ceil_div(kbt, kps);
            u.mtiles = ceil_div(B, BM);
        }
        u.bias_part = b->bpart[l];
        u.wb = b->wb[l];
        u.wt = b->wt[l];
        a.tile0[l - 1] = tiles;
        tiles += (ceil_div(u.n_out, kUT) + 1) * ceil_div(u.n_in, kUT);
    }
    a.tile0[b->L] = tiles;
    a.theta = b->theta;
    a.V = b->V;
    a.G = b->G;
    a.lr_gs = lr_gs;
    a.momentum = momentum;
    a.mode = mode;
    a.fold_g = fold ? 1 : 0;
    a.sse_part = b->sse_part;
    a.n_sse = n_sse;
    a.sse_out = sse_out;
    a.flags = b->flags;
    a.guard = b->guard;
    a.faults = reinterpret_cast<unsigned*>(b->flags + 1);
    return a;
}

cudaError_t launch_update(const UpdArgs& a, int num_sms, cudaStream_t s) {
    int grid = a.tile0[a.L];
    if (grid > num_sms * 8) grid = num_sms * 8;
    if (grid < 1) grid = 1;
    k_update_bf16<<<grid, 256, 0, s>>>(a);
    return cudaGetLastError();
}

}  // namespace

bp_status bf16_check_shape(const int* n, int L, int max_batch) {
    for (int l = 0; l <= L; ++l) {
        if (n[l] % 8 != 0) {
            char buf[200];
            snprintf(buf, sizeof buf,
                     "the bfloat16 path needs every layer size to be a multiple of 8 "
                     "(16-byte rows for TMA); layer %d has %d",
                     l, n[l]);
            g_msg = buf;
            return BP_ESHAPE;
        }
    }
    (void)max_batch;   // transposed copies use a pitch padded to 8; any batch works
    return BP_OK;
}

const char* bf16_last_message() { return g_msg.c_str(); }

bp_status bf16_create(const int* n, int L, int max_batch, int num_sms, float* theta, float* V,
                      float* G, Bf16Net** out) {
    if (!get_encoder()) {
        g_msg = "cuTensorMapEncodeTiled is not available from the driver";
        return BP_ECUDA;
    }
    int dev = 0;
    cudaGetDevice(&dev);
    if (setup_all(dev) != cudaSuccess) {
        g_msg = "could not set the shared-memory limit of the tensor-core kernels";
        return BP_ECUDA;
    }
    Bf16Net* b = new Bf16Net();
    b->L = L;
    for (int l = 0; l <= L; ++l) b->n[l] = n[l];
    b->cap = max_batch;
    b->cap_pad = (max_batch + 7) & ~7;
    b->num_sms = num_sms;
    b->theta = theta;
    b->V = V;
    b->G = G;
    long long pos = 0;
    for (int l = 1; l <= L; ++l) {
        b->woff[l] = pos;
        pos += (long long)n[l] * n[l - 1];
        b->boff[l] = pos;
        pos += n[l];
    }
    bool ok = true;
    const int mt = ceil_div(max_batch, BM);
    for (int l = 0; l <= L && ok; ++l) {
        if (l >= 1) {
            ok = ok && alloc(b, (void**)&b->wb[l], (size_t)n[l] * n[l - 1] * 2);
            ok = ok && alloc(b, (void**)&b->wt[l], (size_t)n[l] * n[l - 1] * 2);
            ok = ok && alloc(b, (void**)&b->act[l], (size_t)max_batch * n[l] * 2);
            ok = ok && alloc(b, (void**)&b->dlt[l], (size_t)max_batch * n[l] * 2);
            ok = ok && alloc(b, (void**)&b->dltT[l], (size_t)n[l] * b->cap_pad * 2);
            const int tiles = ceil_div(n[l], BM) * ceil_div(n[l - 1], kBN);
            b->splits[l] = pick_splits(tiles, ceil_div(max_batch, BK), num_sms, 16);
            ok = ok && alloc(b, (void**)&b->gpart[l], (size_t)b->splits[l] * n[l] * n[l - 1] * 4);
            ok = ok && alloc(b, (void**)&b->bpart[l], (size_t)mt * n[l] * 4);
        }
        if (l < L) ok = ok && alloc(b, (void**)&b->actT[l], (size_t)n[l] * b->cap_pad * 2);
    }
    b->n_sse_cap = mt * ceil_div(n[L], kBN) + mt * ceil_div(n[L], 32);
    ok = ok && alloc(b, (void**)&b->sse_part, (size_t)b->n_sse_cap * 4);
    if (!ok) {
        g_msg = "cudaMalloc failed for the bfloat16 scratch buffers";
        bf16_destroy(b);
        return BP_ENOMEM;
    }
    if (cudaStreamCreateWithFlags(&b->side, cudaStreamNonBlocking) != cudaSuccess ||
        cudaEventCreateWithFlags(&b->fork, cudaEventDisableTiming) != cudaSuccess ||
        cudaEventCreateWithFlags(&b->join, cudaEventDisableTiming) != cudaSuccess) {
        g_msg = "could not create the bfloat16 path's side stream and events";
        bf16_destroy(b);
        return BP_ECUDA;
    }
    *out = b;
    return BP_OK;
}

void bf16_destroy(Bf16Net* b) {
    if (b == nullptr) return;
    if (b->side) cudaStreamSynchronize(b->side);
    if (b->fork) cudaEventDestroy(b->fork);
    if (b->join) cudaEventDestroy(b->join);
    if (b->side) cudaStreamDestroy(b->side);
    for (void* p : b->allocs) cudaFree(p);
    delete b;
}

void bf16_set_flags(Bf16Net* b, int* flags) { b->flags = flags; }
void bf16_set_guard(Bf16Net* b, float guard) { b->guard = guard; }

cudaError_t bf16_refresh_weights(Bf16Net* b, cudaStream_t s) {
    UpdArgs a = upd_args(b, 0, 2, false, 0.f, 0.f, nullptr, 0);
    return launch_update(a, b->num_sms, s);
}

cudaError_t bf16_forward(Bf16Net* b, const void* X, int batch, void* Y, cudaStream_t s) {
    cudaError_t e = run_forward(b, (const bf16*)X, batch, nullptr, b->act[b->L], s);
    if (e != cudaSuccess || Y == nullptr) return e;
    return cudaMemcpy2DAsync(Y, (size_t)b->n[b->L] * 2, b->act[b->L], (size_t)b->n[b->L] * 2,
                             (size_t)b->n[b->L] * 2, batch, cudaMemcpyDeviceToDevice, s);
}

cudaError_t bf16_backward(Bf16Net* b, const void* X, const void* T, int batch, float* sse,
                          bool /*g_dirty*/, cudaStream_t s) {
    const int L = b->L;
    const int nL = b->n[L];
    dim3 grid(ceil_div(nL, 32), ceil_div(batch, 128));
    k_output_delta<<<grid, 128, 0, s>>>(b->act[L], (const bf16*)T, batch, nL, nL, b->dlt[L],
                                        b->dltT[L], b->cap_pad, b->bpart[L], b->sse_part,
                                        ceil_div(nL, 32));
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    e = run_backward(b, (const bf16*)X, batch, s);
    if (e != cudaSuccess) return e;
    UpdArgs a = upd_args(b, batch, 1, false, 0.f, 0.f, sse, ceil_div(batch, 128) * ceil_div(nL, 32));
    return launch_update(a, b->num_sms, s);
}

cudaError_t bf16_update(Bf16Net* b, float lr, float momentum, float grad_scale, cudaStream_t s) {
    // apply G only: no partial changes pending
    UpdArgs a = upd_args(b, 0, 0, true, lr * grad_scale, momentum, nullptr, 0);
    return launch_update(a, b->num_sms, s);
}

cudaError_t bf16_train(Bf16Net* b, const void* X, const void* T, int n_patterns, int minibatch,
                       float* sse, float lr, float momentum, float grad_scale, bool g_dirty,
                       cudaStream_t s) {
    const int L = b->L;
    const size_t xrow = (size_t)b->n[0], trow = (size_t)b->n[L];
    bool fold = g_dirty;
    for (long long p0 = 0, step = 0; p0 < n_patterns; p0 += minibatch, ++step) {
        const int B = (int)((n_patterns - p0) < minibatch ? (n_patterns - p0) : minibatch);
        const bf16* Xs = (const bf16*)X + p0 * xrow;
        const bf16* Ts = (const bf16*)T + p0 * trow;
        cudaError_t e = run_forward(b, Xs, B, Ts, nullptr, s);
        if (e != cudaSuccess) return e;
        e = run_backward(b, Xs, B, s);
        if (e != cudaSuccess) return e;
        const int n_sse = ceil_div(B, BM) * ceil_div(b->n[L], kBN);
        UpdArgs a = upd_args(b, B, 0, fold, lr * grad_scale, momentum,
                             sse != nullptr ? sse + step : nullptr, n_sse);
        e = launch_update(a, b->num_sms, s);
        if (e != cudaSuccess) return e;
        fold = false;
    }
    return cudaSuccess;
}

}  // namespace bp
