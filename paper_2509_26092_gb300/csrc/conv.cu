// conv.cu -- convolution forward, data-gradient and weight-gradient passes of
// ResNet-18 (Sec. 5.1.1; the gradients are those of the batch-mean loss of
// Eq. 1) as implicit GEMMs on the sm_103a tensor cores.
//
// One kernel template serves every pass.  A CTA owns a 128 x BN tile of the
// GEMM result D, accumulated in tensor memory (TMEM) by tcgen05.mma with bf16
// operands and fp32 accumulation:
//
//   pass   D rows (M)          D cols (N)     reduction            A operand            B operand
//   fwd    output pixels n,p,q out channel k  taps x in channels   im2col(x), K-major   w [k][rsc], K-major
//   dgrad  input pixels n,h,w  in channel c   taps x out channels  im2col(dy), K-major  w [k][rs][c], MN-major
//   wgrad  taps x in channel   out channel k  output pixels        im2col(x), MN-major  dy [pix][k], MN-major
//
// Operands are staged in shared memory by TMA: the activation side with
// im2col-mode tensor maps (the bounding box handles zero padding, stride and
// the ragged tail of the last tile), the other side with tiled tensor maps,
// all with 128-byte swizzling (no swizzle for the 8-channel stem input).
// Warp roles: warp 4 issues TMA loads into a STAGES-deep ring guarded by
// full/empty mbarriers, warp 5 allocates TMEM and issues the MMAs (one thread),
// warps 0-3 drain TMEM to global memory (bf16 rows plus BatchNorm channel
// statistics for fwd, fp32 split-K partials for wgrad).
//
// Stride-2 data gradients are split into the 4 output phases (h mod 2,
// w mod 2); each phase is a stride-1 correlation with the taps of matching
// parity, so no MMA work is spent on the zeros of the strided input.
// Every mbarrier wait is bounded (see dbl_internal.cuh); a wait that gives up
// records DBL_ERR_TIMEOUT in the device status word and the CTA winds down.
#include <algorithm>
#include <cstdlib>

#include <atomic>

#include "dbl_internal.cuh"

namespace {

using namespace dbl::dev;

constexpr int BM = 128;        // tile rows = TMEM lanes

enum Mode : int { kFwd = 0, kDgrad = 1, kWgrad = 2, kFwdC8 = 3, kWgradC8 = 4 };

__device__ int g_conv_status;  // DBL_OK or DBL_ERR_TIMEOUT, read by dbl_device_status()

constexpr int kMaxGrid = 256;     // persistent grid never exceeds this (workspace sizing)
constexpr int kMaxNcols = 512;    // widest D (output channels of ResNet-18)

struct ConvParams {
    int mode;
    int M;              // D rows (for dgrad: rows of one phase)
    int Ncols;          // D columns
    int m_tiles, n_tiles, zdim;  // tile grid; zdim = split-K slices (wgrad) or phases (dgrad)
    int total_tiles;
    // traversal grid of the im2col operand: (images, rows, cols) and origin of grid point (0,0)
    int gN, gP, gQ;
    int tstride_h, tstride_w;  // origin step per grid step
    int base_h, base_w;
    int cblocks;        // 64-channel blocks in the reduction (fwd: C/64, dgrad: K/64)
    int ntaps;          // R*S
    int S;              // filter width
    int Cin;            // input channels (fwd B column offset, wgrad row -> (tap, c))
    int num_kb;         // K-blocks of the whole reduction (fwd, wgrad); per phase from the table (dgrad)
    int kb_per_split;   // wgrad split-K chunk
    // dgrad phase tables
    int phase_div;      // 1 or 2
    int out_h, out_w;   // full dx spatial size
    int phase_off[5];
    int8_t tap_r[16], tap_s[16], tap_oh[16], tap_ow[16];
    int proj_kb;        // dgrad phase (0,0): extra K-blocks of a 1x1 stride-2 projection's dy2 . w2
    // outputs
    void* out;          // bf16 rows (fwd, dgrad); fp32 dw (wgrad, one slice) or fp32 slices [z][Ncols][M]
    int64_t ldo;        // elements between output rows (fwd, dgrad)
    int st32;           // 16-bit outputs whose base and row pitch are multiples of 32 bytes: 32-byte stores
    int wg_accumulate;  // wgrad with one slice: add into dw
    float* stats;       // fwd: [gridDim.x][2][Ncols] per-CTA channel sums, or nullptr
    // window kernel (3x3, stride 1, pad 1): the batch as one column of zero-padded images
    int win_R, win_S;         // filter taps along H and W
    int win_ph, win_pw;       // padding along H and W (a strip row copy starts at column -pw)
    int win_P, win_Q;         // output height and width: positions with h < P, w < Q are outputs
    int win_Hp, win_Wp;       // padded height and width (H + 2*ph, W + 2*pw)
    int win_tile;             // positions per tile (weight gradient: per K-block), <= 256
    int win_srows;            // padded rows loaded per strip (weight gradient: x strip)
    int win_dyrows;           // weight gradient: padded rows of the dy strip
    int win_strip_bytes;      // bytes of one strip buffer, or of one x + dy stage (a multiple of 1024)
    int win_margin;           // CTA pairs: bytes before and after each strip buffer (0 for single CTAs)
    int test_stall;           // dbl_conv_test_stall_next: block 0 never loads its first K-block
};

__device__ __forceinline__ void report_timeout(volatile int* abort)
{
    *abort = 1;
    atomicExch(&g_conv_status, DBL_ERR_TIMEOUT);
}

constexpr int kProducers = 2;     // producer warps; producer p fills the stages of iterations it % 2 == p

enum Family : int { kFamFwd = 0, kFamWgrad = 1 };  // fwd/dgrad/stem-fwd, and the two weight-gradient modes

// Per (tile width, family) geometry.  mbarrier round trips and TMA issues cost a
// thread on the order of a hundred cycles each, so every ring stage is sized to
// carry at least ~384 cycles of MMA work per handful of TMA ops:
//   forward family, BN <= 128: a tile is 256 rows in two 128-row accumulators
//     that share one B tile; one 256-pixel im2col op feeds both;
//   weight-gradient family: a K-block is 128 pixels (8 MMA K-steps).
template <int BN, int FAM, int CG = 1>
struct Cfg {
    static constexpr int ACC = (FAM == kFamFwd && BN <= 128) ? 2 : 1;  // 128-row accumulators per tile
    static constexpr int BMT = 128 * ACC;                               // tile rows per CTA
    static constexpr int KB = FAM == kFamFwd ? 64 : 128;                // reduction elements per stage
    static constexpr int KSTEPS = KB / 16;
    static constexpr int BNC = BN / CG;                                 // B columns held by one CTA
    static constexpr int A_BYTES = BMT * KB * 2;
    static constexpr int B_BYTES = BNC * KB * 2;
    static constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
    static constexpr int MAX_STAGES = CG == 2 ? 6 : 4;
    static constexpr int STAGES = (196608 / STAGE_BYTES) < MAX_STAGES ? (196608 / STAGE_BYTES) : MAX_STAGES;
    static constexpr int RING = STAGES * STAGE_BYTES;
    static constexpr int EPI_TILE = 4 * 32 * 33 * 4;           // per-warp 32x32 transpose scratch
    static constexpr int EPI_SUM = 4 * 2 * kMaxNcols * 4;      // per-warp channel sums (fwd)
    static constexpr int SMEM = RING + EPI_TILE + EPI_SUM + 1024;  // + 1 KB alignment slack
    static constexpr int NB = ACC * BN <= 128 ? 4 : 2;          // tiles in flight (TMEM accumulator buffers)
    static constexpr uint32_t TMEM_COLS = NB * ACC * BN;
    static constexpr int THREADS = 32 * (4 + kProducers + 1);   // epilogue, producers, MMA
    static constexpr int MMA_WARP = 4 + kProducers;
    static_assert(STAGES >= 2, "ring too shallow");
    static_assert(TMEM_COLS <= 512, "TMEM holds 512 columns");
    static_assert(SMEM <= 232448 - 1024, "shared memory per CTA");
};

struct TileCoord {
    int m_tile, n_tile, z;
};

// Weight gradient: split-K slice outermost, so that the CTAs running at one time
// share the slice's dy K-blocks.  Stride-2 data gradient: the four phases of one
// m-tile are adjacent, so that the dy rows they all read are fetched from DRAM
// once; the phase index is rotated by one per wave of the persistent grid, so
// that every CTA gets a mix of the 4-, 2- and 1-tap phases.
// units: the number of tiles the persistent grid processes at one time.
__device__ __forceinline__ TileCoord decode_tile(const ConvParams& p, int t, int units)
{
    TileCoord c;
    if (p.mode == kDgrad && p.zdim > 1) {
        const int g = t / p.zdim, l = t - g * p.zdim;
        const int per_wave = max(1, units / p.zdim);
        c.z = (l + g / per_wave) % p.zdim;
        c.m_tile = g / p.n_tiles;
        c.n_tile = g - c.m_tile * p.n_tiles;
        return c;
    }
    const int mn = p.m_tiles * p.n_tiles;
    c.z = t / mn;
    const int r = t - c.z * mn;
    c.m_tile = r / p.n_tiles;
    c.n_tile = r - c.m_tile * p.n_tiles;
    return c;
}

// Number of K-blocks a tile reduces, and the first one.
__device__ __forceinline__ void kb_range(const ConvParams& p, int z, int& kb0, int& nkb)
{
    if (p.mode == kDgrad) {
        kb0 = 0;
        nkb = (p.phase_off[z + 1] - p.phase_off[z]) * p.cblocks + (z == 0 ? p.proj_kb : 0);
    } else if (p.mode == kWgrad || p.mode == kWgradC8) {
        kb0 = z * p.kb_per_split;
        nkb = min(p.num_kb, kb0 + p.kb_per_split) - kb0;
        if (nkb < 0) nkb = 0;
    } else {
        kb0 = 0;
        nkb = p.num_kb;
    }
}

// Issue the TMA loads of one K-block of one tile into ring stage (sa, sb); fb is
// the shared::cluster address of the stage's full barrier.  With CTA pairs
// (CG = 2) CTA `rank` loads its own 128-row (fwd family: BMT-row) part of A and
// columns rank*BN/2 .. (rank+1)*BN/2-1 of B, and both CTAs' loads complete on
// rank 0's barrier.
template <int BN, int FAM, int CG>
__device__ __forceinline__ void load_kblock(const ConvParams& p, const CUtensorMap* tmA, const CUtensorMap* tmB,
                                            const CUtensorMap* tmA2, const CUtensorMap* tmB2, uint8_t* sa,
                                            uint8_t* sb, uint32_t fb, const TileCoord& tc, int kb, int tn, int tp,
                                            int tq, int rank)
{
    using C = Cfg<BN, FAM, CG>;
    const int64_t gPQ = (int64_t)p.gP * p.gQ;
    const int ncol0 = tc.n_tile * BN + rank * C::BNC;  // first B column this CTA loads
    if constexpr (FAM == kFamFwd) {
        if (p.mode == kFwd) {
            const int tap = kb / p.cblocks, cb = kb - tap * p.cblocks;
            const int r = tap / p.S, sx = tap - r * p.S;
            tma_load_im2col_4d_cg<CG>(sa, tmA, fb, cb * 64, tq * p.tstride_w + p.base_w, tp * p.tstride_h + p.base_h, tn,
                                      (uint16_t)sx, (uint16_t)r);
            tma_load_2d_cg<CG>(sb, tmB, fb, tap * p.Cin + cb * 64, ncol0);
        } else if (p.mode == kDgrad && kb >= (p.phase_off[tc.z + 1] - p.phase_off[tc.z]) * p.cblocks) {
            // phase (0,0) of a stride-2 data gradient with a 1x1 stride-2 projection shortcut on
            // the same input: dx[n, 2i, 2j] also receives dy2[n, i, j] . w2, the dy2 rows of this
            // tile being the tile's own rows m0.. (tmA2: dy2 as [n*P*Q][k2], tmB2: w2 as [k2][1][c])
            const int e = kb - (p.phase_off[tc.z + 1] - p.phase_off[tc.z]) * p.cblocks;
            const int m0 = (tn * p.gP + tp) * p.gQ + tq;
            tma_load_2d_cg<CG>(sa, tmA2, fb, e * 64, m0);
            for (int j = 0; j < C::BNC / 64; ++j) tma_load_3d_cg<CG>(sb + j * 8192, tmB2, fb, ncol0 + 64 * j, 0, e * 64);
        } else if (p.mode == kDgrad) {
            const int t = p.phase_off[tc.z] + kb / p.cblocks, kbk = kb % p.cblocks;
            tma_load_im2col_4d_cg<CG>(sa, tmA, fb, kbk * 64, tq + p.base_w, tp + p.base_h, tn, (uint16_t)p.tap_ow[t],
                                      (uint16_t)p.tap_oh[t]);
            const int wtap = p.tap_r[t] * p.S + p.tap_s[t];
            for (int j = 0; j < C::BNC / 64; ++j)
                tma_load_3d_cg<CG>(sb + j * 8192, tmB, fb, ncol0 + 64 * j, wtap, kbk * 64);
        } else {  // kFwdC8: 8 taps of 8 channels; taps past R*S read a valid tap and meet zero weights
            for (int j = 0; j < 8; ++j) {
                int tap = kb * 8 + j;
                const int wcol = tap * 8;
                if (tap >= p.ntaps) tap = p.ntaps - 1;
                tma_load_im2col_4d_cg<CG>(sa + j * (C::BMT * 16), tmA, fb, 0, tq * p.tstride_w + p.base_w,
                                          tp * p.tstride_h + p.base_h, tn, (uint16_t)(tap % p.S), (uint16_t)(tap / p.S));
                tma_load_2d_cg<CG>(sb + j * (C::BNC * 16), tmB, fb, wcol, ncol0);
            }
        }
    } else {
        // weight gradient: a K-block is 128 output pixels
        const int64_t pix0 = (int64_t)kb * 128;
        const int n = (int)(pix0 / gPQ);
        const int64_t rem = pix0 - (int64_t)n * gPQ;
        const int pp = (int)(rem / p.gQ), qq = (int)(rem - (int64_t)pp * p.gQ);
        if (p.mode == kWgrad) {
            for (int h = 0; h < 2; ++h) {
                const int mrow = (tc.m_tile * CG + rank) * BM + 64 * h;
                int tap = mrow / p.Cin;
                const int c0 = mrow - tap * p.Cin;
                if (tap >= p.ntaps) tap = 0;  // rows past R*S*C: loaded, never stored
                tma_load_im2col_4d_cg<CG>(sa + h * 16384, tmA, fb, c0, qq * p.tstride_w + p.base_w,
                                          pp * p.tstride_h + p.base_h, n, (uint16_t)(tap % p.S), (uint16_t)(tap / p.S));
            }
        } else {  // kWgradC8: 16 taps x 8 channels of rows
            for (int j = 0; j < 16; ++j) {
                int tap = tc.m_tile * 16 + j;
                if (tap >= p.ntaps) tap = 0;
                tma_load_im2col_4d_cg<CG>(sa + j * 2048, tmA, fb, 0, qq * p.tstride_w + p.base_w,
                                          pp * p.tstride_h + p.base_h, n, (uint16_t)(tap % p.S), (uint16_t)(tap / p.S));
            }
        }
        for (int j = 0; j < C::BNC / 64; ++j) tma_load_2d_cg<CG>(sb + j * 16384, tmB, fb, ncol0 + 64 * j, (int)pix0);
    }
}

// Epilogue of the 16-bit-output passes for one 32-column chunk of this thread's
// accumulator row: round to the storage format (bf16, or f16) and store the row chunk (if the row is a real
// output); back[] receives the stored values (zeros for rows that are not outputs).
__device__ __forceinline__ void store_row_chunk_act(const ConvParams& p, const uint32_t (&v)[32], bool valid,
                                                     int64_t out_row, int col0, float (&back)[32])
{
    uint4 pk[4];
    uint32_t* w32 = reinterpret_cast<uint32_t*>(pk);
#pragma unroll
    for (int k = 0; k < 16; ++k) {
        const uint32_t u = valid ? dbl::act::pack2_u32(__uint_as_float(v[2 * k]), __uint_as_float(v[2 * k + 1]))
                                 : 0u;  // rows that are not outputs: 0
        w32[k] = u;
        const float2 f = dbl::act::unpack2_u32(u);  // the stored values (16-bit -> fp32 is exact)
        back[2 * k] = f.x;
        back[2 * k + 1] = f.y;
    }
    if (valid) {
        act_t* o = static_cast<act_t*>(p.out) + out_row * p.ldo + col0;
        if (p.st32) {
            // whole 32-byte sectors per instruction: half the store instructions and L2 write
            // requests of 16-byte stores, each of which fills half a sector
#pragma unroll
            for (int k = 0; k < 2; ++k)
                asm volatile("st.global.v8.b32 [%0], {%1, %2, %3, %4, %5, %6, %7, %8};" ::"l"(o + 16 * k),
                             "r"(pk[2 * k].x), "r"(pk[2 * k].y), "r"(pk[2 * k].z), "r"(pk[2 * k].w),
                             "r"(pk[2 * k + 1].x), "r"(pk[2 * k + 1].y), "r"(pk[2 * k + 1].z), "r"(pk[2 * k + 1].w)
                             : "memory");
        } else {
#pragma unroll
            for (int k = 0; k < 4; ++k) reinterpret_cast<uint4*>(o)[k] = pk[k];
        }
    }
}

// BatchNorm channel sums (sum y, sum y^2) of the stored forward outputs, kept
// in registers across the tiles of a CTA instead of being reduced across the
// warp for every tile (which costs shared-memory bandwidth that the mainloop
// needs).  Thread (warp, lane) adds the values of its own accumulator row.
// For BN > 64 the rows are first folded pairwise across lanes (LEVELS
// shuffle steps), so that every thread holds 128 sums: after the folding,
// value k of chunk ch belongs to column ch*32 + (lane & (32 - V)) + k.
// flush() reduces over the lanes through the warp's 32x33 scratch and adds the
// column totals to the warp's channel sums (once per CTA, and whenever the
// CTA moves to another column tile).
template <int BN>
struct RowStats {
    static constexpr int NCH = BN / 32;
    static constexpr int LEVELS = BN <= 64 ? 0 : (BN <= 128 ? 1 : 2);
    static constexpr int V = 32 >> LEVELS;
    float s[NCH][V], q[NCH][V];

    __device__ __forceinline__ void zero()
    {
#pragma unroll
        for (int c = 0; c < NCH; ++c)
#pragma unroll
            for (int k = 0; k < V; ++k) s[c][k] = q[c][k] = 0.f;
    }

    template <int N, int O>
    __device__ __forceinline__ static void fold(float (&a)[32], float (&b)[32], int lane)
    {
        const bool up = (lane & O) != 0;
#pragma unroll
        for (int k = 0; k < N / 2; ++k) {
            const float sa = up ? a[k] : a[k + N / 2], ka = up ? a[k + N / 2] : a[k];
            const float sb = up ? b[k] : b[k + N / 2], kb = up ? b[k + N / 2] : b[k];
            a[k] = ka + __shfl_xor_sync(0xffffffffu, sa, O);
            b[k] = kb + __shfl_xor_sync(0xffffffffu, sb, O);
        }
    }

    // x: the stored values of chunk ch of this thread's row (call with ch a compile-time
    // constant after unrolling).  Every lane of the warp must call it.
    __device__ __forceinline__ void add(int ch, const float (&x)[32], int lane)
    {
        if constexpr (LEVELS == 0) {  // no folding: sum of squares by fused multiply-add
#pragma unroll
            for (int k = 0; k < 32; ++k) {
                s[ch][k] += x[k];
                q[ch][k] = fmaf(x[k], x[k], q[ch][k]);
            }
        } else {
            float a[32], b[32];
#pragma unroll
            for (int k = 0; k < 32; ++k) {
                a[k] = x[k];
                b[k] = x[k] * x[k];
            }
            if constexpr (LEVELS >= 1) fold<32, 16>(a, b, lane);
            if constexpr (LEVELS >= 2) fold<16, 8>(a, b, lane);
#pragma unroll
            for (int k = 0; k < V; ++k) {
                s[ch][k] += a[k];
                q[ch][k] += b[k];
            }
        }
    }

    // wsum: this warp's [2][Ncols] channel sums; col_base: first column of the tile.
    __device__ __forceinline__ void flush(float* st_tile, float* wsum, int ncols, int col_base, int lane)
    {
        const int hb = lane & (32 - V), kk = lane & (V - 1);
#pragma unroll
        for (int c = 0; c < NCH; ++c) {
#pragma unroll
            for (int w = 0; w < 2; ++w) {
#pragma unroll
                for (int k = 0; k < V; ++k) st_tile[lane * 33 + k] = w ? q[c][k] : s[c][k];
                __syncwarp();
                float tot = 0.f;
#pragma unroll
                for (int u = 0; u < V; ++u) tot += st_tile[(hb + u) * 33 + kk];
                __syncwarp();
                wsum[w * ncols + col_base + c * 32 + lane] += tot;
            }
        }
        zero();
    }
};

// Persistent kernel: CTA b processes tiles b, b + gridDim.x, ...  The ring of
// STAGES shared-memory stages runs continuously across tiles; two producer
// warps fill alternate stages; two TMEM accumulators let the epilogue of one
// tile overlap the MMAs of the next.
//
// CG = 2 (clusters of two CTAs): a tile is processed by a CTA pair with
// M = 256 MMAs (tcgen05 .cta_group::2).  Each CTA stages its own BMT rows of A
// and half of the B columns, so a CTA's shared memory carries half of the B
// bytes (TMA writes and MMA reads) of the single-CTA form; shared-memory
// bandwidth is what limits the single-CTA form.  Rank 0 issues the MMAs and owns
// the stage-full barriers, which both CTAs' loads complete on; its commits
// arrive on the stage-empty and accumulator-full barriers of both CTAs; the
// epilogues of both CTAs arrive on rank 0's accumulator-empty barriers.  Each
// CTA drains its own TMEM (its own rows, all BN columns).
template <int BN, int FAM, int CG>
__global__ void __launch_bounds__(Cfg<BN, FAM, CG>::THREADS, 1)
    conv_igemm_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                      const __grid_constant__ CUtensorMap tmA2, const __grid_constant__ CUtensorMap tmB2,
                      const ConvParams p)
{
    dbl::dev::grid_dependency_trigger();  // a convolution launched next may start its set-up
    using C = Cfg<BN, FAM, CG>;
    constexpr int STAGES = C::STAGES;
    extern __shared__ uint8_t smem_raw[];
    __shared__ __align__(8) uint64_t full_bar[STAGES], empty_bar[STAGES], accf_bar[C::NB], acce_bar[C::NB], drain_bar;
    __shared__ uint32_t tmem_slot;
    __shared__ volatile int abort_flag;

    const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
    const uint32_t sbase = (smem_u32(smem_raw) + 1023u) & ~1023u;
    uint8_t* sgen = smem_raw + (sbase - smem_u32(smem_raw));
    float* epi_tile = reinterpret_cast<float*>(sgen + C::RING);
    float* epi_sum = reinterpret_cast<float*>(sgen + C::RING + C::EPI_TILE);
    const int rank = CG == 2 ? (int)cluster_ctarank() : 0;
    const int unit0 = blockIdx.x / CG, nunits = gridDim.x / CG;  // this pair's first tile, tiles' stride

    if (threadIdx.x == 0) {
        for (int s = 0; s < STAGES; ++s) {
            mbar_init(&full_bar[s], 1);
            mbar_init(&empty_bar[s], 1);
        }
        for (int b = 0; b < C::NB; ++b) {
            mbar_init(&accf_bar[b], 1);
            mbar_init(&acce_bar[b], 4 * CG);  // one arrival per epilogue warp of the pair
        }
        mbar_init(&drain_bar, 1);
        abort_flag = 0;
        fence_mbar_init();
    }
    const bool want_stats = FAM == kFamFwd && (p.mode == kFwd || p.mode == kFwdC8) && p.stats != nullptr;
    if (want_stats)
        for (int i = threadIdx.x; i < 4 * 2 * p.Ncols; i += blockDim.x) epi_sum[i] = 0.f;
    if (warp >= 4 && warp < 4 + kProducers && lane == 0) {
        tma_prefetch_desc(&tmA);
        tma_prefetch_desc(&tmB);
        if (p.proj_kb) {
            tma_prefetch_desc(&tmA2);
            tma_prefetch_desc(&tmB2);
        }
    }
    if (warp == C::MMA_WARP) {
        tmem_alloc_cg<CG>(&tmem_slot, C::TMEM_COLS);
        tmem_relinquish_cg<CG>();
    }
    tc_fence_before();
    __syncthreads();
    if constexpr (CG == 2) cluster_sync_all();  // both CTAs' barriers initialised, TMEM allocated
    tc_fence_after();
    grid_dependency_wait();  // the set-up above may overlap the previous kernel; memory only after it
    const uint32_t tmem = tmem_slot;
    const int64_t gPQ = (int64_t)p.gP * p.gQ;

    if (warp >= 4 && warp < 4 + kProducers) {
        // ------------------------------------------------------------------ TMA producers (whole warp, one lane issues)
        const int prod = warp - 4;
        int it = 0, last_it = -1;
        bool failed = false;
        for (int t = unit0; t < p.total_tiles; t += nunits) {
            const TileCoord tc = decode_tile(p, t, nunits);
            int kb0, nkb;
            kb_range(p, tc.z, kb0, nkb);
            int tn = 0, tp = 0, tq = 0;
            if (FAM == kFamFwd) {
                const int64_t m0 = ((int64_t)tc.m_tile * CG + rank) * C::BMT;
                tn = (int)(m0 / gPQ);
                const int64_t rem = m0 - (int64_t)tn * gPQ;
                tp = (int)(rem / p.gQ);
                tq = (int)(rem - (int64_t)tp * p.gQ);
            }
            for (int k = 0; k < nkb; ++k, ++it) {
                if (it % kProducers != prod) continue;
                if (p.test_stall && blockIdx.x == 0 && it == 0) continue;  // stage 0 never fills (bounded-wait test)
                const int s = it % STAGES;
                const uint32_t ok = mbar_wait_warp(&empty_bar[s], ((it / STAGES) & 1) ^ 1, &abort_flag);
                if (__any_sync(0xffffffffu, ok == 0u)) {
                    failed = true;
                    break;
                }
                uint8_t* sa = sgen + s * C::STAGE_BYTES;
                uint32_t fb = smem_u32(&full_bar[s]);
                if (CG == 1 || rank == 0)
                    mbar_arrive_expect_tx_elect(&full_bar[s], (uint32_t)(CG * C::STAGE_BYTES));
                if (CG == 2) fb = mapa_shared(fb, 0);
                load_kblock<BN, FAM, CG>(p, &tmA, &tmB, &tmA2, &tmB2, sa, sa + C::A_BYTES, fb, tc, kb0 + k, tn, tp, tq,
                                         rank);
                last_it = it;
            }
            if (failed) break;
        }
        if (failed) {
            if (lane == 0) report_timeout(&abort_flag);
            if (CG == 1 || rank == 0) {
                // let copies this producer issued land before the CTA's shared memory goes away
                for (int i = last_it; i >= 0 && i > last_it - STAGES * kProducers; i -= kProducers)
                    (void)mbar_drain_warp(&full_bar[i % STAGES], (i / STAGES) & 1);
            } else {
                // rank 1's copies complete on rank 0's barriers: give them a fixed time instead
                const uint64_t t0 = globaltimer();
                while (globaltimer() - t0 < 1000000ull) {
                }
            }
        }
    } else if (warp == C::MMA_WARP) {
        // ------------------------------------------------------------------ MMA issuer (whole warp, one lane issues)
        const bool a_mn = (p.mode == kWgrad || p.mode == kWgradC8);
        const bool b_mn = (p.mode != kFwd && p.mode != kFwdC8);
        const uint32_t idesc = idesc_act(BM * CG, BN, a_mn ? 1u : 0u, b_mn ? 1u : 0u);
        constexpr uint16_t kAll = CG == 2 ? 3 : 1;  // commits reach both CTAs of a pair
        // Operand descriptors without their start address, and the start-address steps
        // (in 16-byte units) per K-step and per accumulator:
        //   kFwd / kDgrad: A K-major, 128-byte swizzle, one K-step = 32 bytes of a row;
        //     B K-major (fwd) or MN-major with 64-wide atoms 8 KB apart (dgrad, 2 KB per K-step);
        //   kFwdC8: K-major without swizzle: core matrices of 8 rows x 16 B, rows 16 B apart,
        //     8-row groups 128 B apart (SBO), the two taps of one K-step LBO apart;
        //   kWgrad: both MN-major, 128-byte swizzle, 64-wide atoms 16 KB apart (LBO);
        //   kWgradC8: A MN-major without swizzle, 8 pixels x 8 channels per core matrix,
        //     next 8 pixels 128 B apart (LBO), next tap 2 KB apart (SBO).
        uint64_t dA, dB;
        int a_step16, b_step16, a_acc16 = 16384 / 16;
        if (p.mode == kFwd || p.mode == kDgrad) {
            dA = smem_desc(0, 16, 1024, kSwizzle128B);
            a_step16 = 2;
            if (p.mode == kFwd) {
                dB = smem_desc(0, 16, 1024, kSwizzle128B);
                b_step16 = 2;
            } else {
                dB = smem_desc(0, 8192, 1024, kSwizzle128B);
                b_step16 = 2048 / 16;
            }
        } else if (p.mode == kFwdC8) {
            dA = smem_desc(0, C::BMT * 16, 128, kSwizzleNone);
            dB = smem_desc(0, C::BNC * 16, 128, kSwizzleNone);
            a_step16 = 2 * C::BMT;
            b_step16 = 2 * C::BNC;
            a_acc16 = 2048 / 16;
        } else if (p.mode == kWgrad) {
            dA = smem_desc(0, 16384, 1024, kSwizzle128B);
            dB = smem_desc(0, 16384, 1024, kSwizzle128B);
            a_step16 = b_step16 = 2048 / 16;
        } else {
            dA = smem_desc(0, 128, 2048, kSwizzleNone);
            dB = smem_desc(0, 16384, 1024, kSwizzle128B);
            a_step16 = 256 / 16;
            b_step16 = 2048 / 16;
        }
        // The MMA issue is on the critical path: every cycle this warp spends polling a
        // barrier while the tensor pipe has nothing queued is lost.  So the wait for the next
        // stage is made before the last K-step of the current stage is issued, while the
        // tensor pipe still has work.
        bool failed = false;
        auto wait_ok = [&](uint64_t* bar, uint32_t parity) -> bool {
            const uint32_t ok = mbar_wait_warp(bar, parity, &abort_flag);
            return !__any_sync(0xffffffffu, ok == 0u);
        };
        // Only waits inside a tile are made ahead: waiting for the next tile's accumulator or
        // data before this tile's last K-step would delay this tile's completion, and with it
        // the epilogue, behind an earlier epilogue or a later load.
        int it = 0, lt = 0;
        for (int t = unit0; t < p.total_tiles && (CG == 1 || rank == 0) && !failed; t += nunits, ++lt) {
            const TileCoord tc = decode_tile(p, t, nunits);
            int kb0, nkb;
            kb_range(p, tc.z, kb0, nkb);
            const int buf = lt % C::NB;
            if (!wait_ok(&acce_bar[buf], ((lt / C::NB) & 1) ^ 1) ||
                (nkb > 0 && !wait_ok(&full_bar[it % STAGES], (it / STAGES) & 1))) {
                failed = true;
                break;
            }
            const uint32_t d = tmem + (uint32_t)(buf * C::ACC * BN);
            for (int k = 0; k < nkb; ++k, ++it) {
                tc_fence_after();
                const int s = it % STAGES;
                const uint32_t sa = sbase + s * C::STAGE_BYTES;
                const uint32_t sb = sa + C::A_BYTES;
                const uint64_t ad0 = dA | (uint64_t)((sa >> 4) & 0x3FFFu), bd0 = dB | (uint64_t)((sb >> 4) & 0x3FFFu);
#pragma unroll
                for (int j = 0; j < C::KSTEPS - 1; ++j) {
#pragma unroll
                    for (int a = 0; a < C::ACC; ++a)
                        mma_act_elect_cg<CG>(d + a * BN, ad0 + (uint64_t)(a * a_acc16 + j * a_step16),
                                              bd0 + (uint64_t)(j * b_step16), idesc, (k > 0 || j > 0) ? 1u : 0u);
                }
                if (k + 1 < nkb) failed = !wait_ok(&full_bar[(it + 1) % STAGES], ((it + 1) / STAGES) & 1);
                constexpr int jl = C::KSTEPS - 1;
#pragma unroll
                for (int a = 0; a < C::ACC; ++a)
                    mma_act_elect_cg<CG>(d + a * BN, ad0 + (uint64_t)(a * a_acc16 + jl * a_step16),
                                          bd0 + (uint64_t)(jl * b_step16), idesc, (k > 0 || jl > 0) ? 1u : 0u);
                mma_commit_elect_cg<CG>(&empty_bar[s], kAll);
                if (failed) {
                    ++it;
                    break;
                }
            }
            mma_commit_elect_cg<CG>(&accf_bar[buf], kAll);  // arrives when this tile's MMAs have completed
        }
        if (failed && lane == 0) report_timeout(&abort_flag);
        if (CG == 1 || rank == 0) {
            // every MMA issued above completes before the accumulators are freed
            mma_commit_elect_cg<CG>(&drain_bar, 1);
            (void)mbar_drain_warp(&drain_bar, 0);
        }
    } else {
        // ------------------------------------------------------------------ epilogue (warps 0-3)
        float* st_tile = epi_tile + warp * 32 * 33;
        float* wsum = epi_sum + warp * 2 * p.Ncols;
        RowStats<BN> rs;
        rs.zero();
        int stats_ntile = -1;  // column tile the register sums belong to
        int lt = 0;
        for (int t = unit0; t < p.total_tiles; t += nunits, ++lt) {
            const TileCoord tc = decode_tile(p, t, nunits);
            int kb0, nkb;
            kb_range(p, tc.z, kb0, nkb);
            const int buf = lt % C::NB;
            const uint32_t ok = mbar_wait_warp(&accf_bar[buf], (lt / C::NB) & 1, &abort_flag);
            if (__any_sync(0xffffffffu, ok == 0u)) {
                if (lane == 0) report_timeout(&abort_flag);
                break;
            }
            tc_fence_after();
            const int row = warp * 32 + lane;  // TMEM lane = row within a 128-row accumulator
            const bool have_acc = nkb > 0;
            if (want_stats && stats_ntile != tc.n_tile) {
                if (stats_ntile >= 0) rs.flush(st_tile, wsum, p.Ncols, stats_ntile * BN, lane);
                stats_ntile = tc.n_tile;
            }
#pragma unroll 1
            for (int a = 0; a < C::ACC; ++a) {
                const int64_t m = ((int64_t)tc.m_tile * CG + rank) * C::BMT + a * 128 + row;
                const bool valid = m < p.M;
                const uint32_t taddr = tmem + ((uint32_t)(warp * 32) << 16) + (uint32_t)((buf * C::ACC + a) * BN);
                if constexpr (FAM == kFamWgrad) {
#pragma unroll 1
                    for (int ch = 0; ch < BN / 32; ++ch) {
                        uint32_t v[32];
                        if (have_acc) {
                            tmem_ld_32x32b_x32(taddr + ch * 32, v);
                            tmem_ld_wait();
                        } else {
#pragma unroll
                            for (int k = 0; k < 32; ++k) v[k] = 0u;
                        }
                        const int col0 = tc.n_tile * BN + ch * 32;
                        // D row m = (tap, c), column = output channel k; stored as [slice][k][m]:
                        // consecutive lanes hold consecutive m, so each store is one 128-byte line
                        if (valid) {
                            float* o = static_cast<float*>(p.out) + ((int64_t)tc.z * p.Ncols + col0) * p.M + m;
                            if (p.zdim == 1 && p.wg_accumulate) {
#pragma unroll
                                for (int k = 0; k < 32; ++k) o[(int64_t)k * p.M] += __uint_as_float(v[k]);
                            } else {
#pragma unroll
                                for (int k = 0; k < 32; ++k) o[(int64_t)k * p.M] = __uint_as_float(v[k]);
                            }
                        }
                    }
                } else {
                    int64_t out_row = m;
                    if (p.mode == kDgrad && p.phase_div == 2) {
                        const int64_t n = m / gPQ, rem = m - n * gPQ;
                        const int i = (int)(rem / p.gQ), j = (int)(rem - (int64_t)(rem / p.gQ) * p.gQ);
                        const int pa = tc.z >> 1, pb = tc.z & 1;
                        out_row = (n * p.out_h + 2 * i + pa) * p.out_w + 2 * j + pb;
                    }
#pragma unroll
                    for (int ch = 0; ch < BN / 32; ++ch) {
                        uint32_t v[32];
                        if (have_acc) {
                            tmem_ld_32x32b_x32(taddr + ch * 32, v);
                            tmem_ld_wait();
                        } else {
#pragma unroll
                            for (int k = 0; k < 32; ++k) v[k] = 0u;
                        }
                        float back[32];
                        store_row_chunk_act(p, v, valid, out_row, tc.n_tile * BN + ch * 32, back);
                        if (want_stats) rs.add(ch, back, lane);
                    }
                }
            }
            tc_fence_before();
            __syncwarp();
            if (lane == 0) {
                if constexpr (CG == 2)
                    mbar_arrive_cluster(mapa_shared(smem_u32(&acce_bar[buf]), 0));
                else
                    mbar_arrive(&acce_bar[buf]);
            }
        }
        if (want_stats && stats_ntile >= 0) rs.flush(st_tile, wsum, p.Ncols, stats_ntile * BN, lane);
        if (want_stats) {
            asm volatile("bar.sync 1, 128;" ::: "memory");
            float* dst = p.stats + (int64_t)blockIdx.x * 2 * p.Ncols;
            for (int c = threadIdx.x; c < 2 * p.Ncols; c += 128)
                dst[c] = (epi_sum[c] + epi_sum[2 * p.Ncols + c]) + (epi_sum[4 * p.Ncols + c] + epi_sum[6 * p.Ncols + c]);
        }
    }
    tc_fence_before();
    __syncthreads();
    // neither CTA of a pair leaves while the other may still signal its barriers or read its TMEM
    if constexpr (CG == 2) cluster_sync_all();
    if (warp == C::MMA_WARP) {
        tc_fence_after();
        tmem_dealloc_cg<CG>(tmem, C::TMEM_COLS);
    }
}

// ----------------------------------------------------------------------------- window kernel
// 3x3, stride-1, pad-1 correlation (the forward pass, and the data gradient
// with the taps flipped) without im2col.  Position (h, w) of image n of the
// zero-padded input is row g = n*Hp + h of a column of padded rows, and
// padded position L = g*Wp + w.  Output (h, w) of image n is computed at
// L = (n*Hp + h)*Wp + w, and its tap (r, s) reads padded position L + r*Wp + s.
// So a tile of 256 consecutive L needs one strip of padded rows (TMA loads
// one padded row per copy: the box starts at w = -1 and the zero fill makes
// the padding), and each of the nine taps is the same strip addressed by a
// descriptor that starts r*Wp + s rows later.  The 128-byte swizzle of both
// TMA and the MMA operand fetch is a function of the absolute shared-memory
// address, so a start at any 128-byte row reads the rows that TMA wrote.  Rows
// with h >= H or w >= W are computed and not stored (the padding's share of
// the work: 7% at 56x56, 13% at 28x28).
// Warp roles: warp 4 loads strips (two buffers), warp 5 loads weights (all
// nine taps once per CTA when they fit, RES; else a ring of per-tap tiles),
// warp 6 issues the MMAs, warps 0-3 drain TMEM as in conv_igemm_kernel.
constexpr int kWinACC = 2;               // 128-row accumulators per tile
constexpr int kWinBMT = 128 * kWinACC;   // padded positions per tile
constexpr int kWinBStages = 4;           // weight-tile ring depth when not resident
constexpr int kWinThreads = 224;         // conv_wgwin_kernel: 4 epilogue warps, 2 producers, MMA

// Warp roles of conv_win_kernel: EPI epilogue warps (0 .. EPI-1), then the strip
// producer, the weight producer and the MMA issuer.  (Eight epilogue warps, two per
// TMEM lane quarter, and stores staged in shared memory so that each instruction
// writes whole lines, both measured slower on the stem than this form.)
template <int BN>
struct WinCfg {
    static constexpr int B_TILE = BN * 64 * 2;  // one tap x one 64-channel block of weights
    static constexpr int NB = BN == 64 ? 4 : 2;  // accumulator buffers (tiles in flight)
    static constexpr uint32_t TMEM_COLS = NB * kWinACC * BN;
    static constexpr int EPI = 4;                // epilogue warps
    static constexpr int CW = BN * 4 / EPI;      // columns one epilogue warp drains
    static constexpr int W_STRIP = EPI, W_WEIGHT = EPI + 1, W_MMA = EPI + 2;
    static constexpr int THREADS = 32 * (EPI + 3);
};

// One tap x 64-channel block of weights: K-major [BN out][64 in] for the forward
// pass, MN-major [64 k][BN c] blocks of 64 for the data gradient (flipped tap).
// CG = 2: this CTA's half of the BN columns (rank r: columns r*BN/2 ..), completing
// on the barrier at shared::cluster address bar (the leader's).
template <int BN, bool DG, int CG>
__device__ __forceinline__ void win_load_wtile(const ConvParams& p, const CUtensorMap* tmB, uint8_t* dst, uint32_t bar,
                                               int tap, int cb, int n_tile, int rank)
{
    if constexpr (DG) {
        const int wtap = p.win_R * p.win_S - 1 - tap;  // flipped filter
#pragma unroll
        for (int j = 0; j < BN / 64 / CG; ++j)
            tma_load_3d_cg<CG>(dst + j * 8192, tmB, bar, n_tile * BN + rank * (BN / CG) + 64 * j, wtap, cb * 64);
    } else {
        tma_load_2d_cg<CG>(dst, tmB, bar, tap * p.Cin + cb * 64, n_tile * BN + rank * (BN / CG));
    }
}

// CG = 2 (a cluster of two CTAs, tcgen05 .cta_group::2): CTA rank r computes tile
// 2u + r of pair unit u.  Rank 0 issues M = 256 MMAs whose A rows 0-127 come from
// its strip and rows 128-255 from rank 1's, at the same shared-memory address, and
// whose B columns are split between the two CTAs' halves of the weights, so each SM
// reads half of B per MMA.  The two tiles start at different offsets within a
// padded row (off0), so rank 1 places its strip (off0 of rank 0 - off0 of rank 1)
// rows away from rank 0's (inside a margin of one padded row on either side): the
// descriptors rank 0 builds from its own off0 then read rank 1's tile at the same
// rows.  Rank 0 owns the strip-full, weight-full and accumulator-empty barriers;
// both CTAs' copies complete on rank 0's full barriers, rank 0's commits arrive on
// both CTAs' empty and accumulator-full barriers, and both CTAs' epilogues arrive on
// rank 0's accumulator-empty barrier.  A pair unit past the last tile loads zeros
// (images past the batch) and stores nothing.
template <int BN, bool DG, bool RES, int CG>
__global__ void __launch_bounds__(WinCfg<BN>::THREADS, 1)
    conv_win_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                    const ConvParams p)
{
    dbl::dev::grid_dependency_trigger();  // a convolution launched next may start its set-up
    using C = WinCfg<BN>;
    static_assert(CG == 1 || BN == 128 || !DG, "data-gradient pairs split the weights in 64-column halves");
    constexpr int BT = C::B_TILE / CG;  // this CTA's bytes of one tap x 64-channel block of weights
    constexpr uint16_t kAll = CG == 2 ? 3 : 1;
    extern __shared__ uint8_t smem_raw[];
    __shared__ __align__(8) uint64_t sfull[2], sempty[2], bfull[kWinBStages], bempty[kWinBStages], accf_bar[4],
        acce_bar[4], drain_bar;
    __shared__ uint32_t tmem_slot;
    __shared__ volatile int abort_flag;

    const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
    const uint32_t sbase = (smem_u32(smem_raw) + 1023u) & ~1023u;
    uint8_t* sgen = smem_raw + (sbase - smem_u32(smem_raw));
    const int rank = CG == 2 ? (int)cluster_ctarank() : 0;
    const int unit0 = blockIdx.x / CG, nunits = gridDim.x / CG;
    const int total_units = (p.total_tiles + CG - 1) / CG;
    const int CB = p.cblocks;
    const int ntaps = p.win_R * p.win_S;
    const int b_bytes = RES ? ntaps * CB * BT : kWinBStages * BT;
    const int strip_stride = p.win_strip_bytes + 2 * p.win_margin;
    uint8_t* strip = sgen + b_bytes + p.win_margin;  // stage s at strip + s * strip_stride
    // per-warp statistics transposes reuse the strip buffers once the last tile's MMAs are done
    float* epi_tile = reinterpret_cast<float*>(sgen + b_bytes);
    float* epi_sum = reinterpret_cast<float*>(sgen + b_bytes + 2 * strip_stride);

    if (threadIdx.x == 0) {
        for (int i = 0; i < 2; ++i) {
            mbar_init(&sfull[i], 1);
            mbar_init(&sempty[i], 1);
        }
        for (int i = 0; i < C::NB; ++i) {
            mbar_init(&accf_bar[i], 1);
            mbar_init(&acce_bar[i], C::EPI * CG);  // one arrival per epilogue warp of the pair
        }
        for (int i = 0; i < kWinBStages; ++i) {
            mbar_init(&bfull[i], 1);
            mbar_init(&bempty[i], 1);
        }
        mbar_init(&drain_bar, 1);
        abort_flag = 0;
        fence_mbar_init();
    }
    const bool want_stats = p.mode == kFwd && p.stats != nullptr;
    if (want_stats)
        for (int i = threadIdx.x; i < C::EPI * 2 * p.Ncols; i += blockDim.x) epi_sum[i] = 0.f;
    if ((warp == C::W_STRIP || warp == C::W_WEIGHT) && lane == 0) {
        tma_prefetch_desc(&tmA);
        tma_prefetch_desc(&tmB);
    }
    if (warp == C::W_MMA) {
        tmem_alloc_cg<CG>(&tmem_slot, C::TMEM_COLS);
        tmem_relinquish_cg<CG>();
    }
    tc_fence_before();
    __syncthreads();
    if constexpr (CG == 2) cluster_sync_all();  // both CTAs' barriers initialised, TMEM allocated
    tc_fence_after();
    grid_dependency_wait();  // the set-up above may overlap the previous kernel; memory only after it
    const uint32_t tmem = tmem_slot;
    const int Wp = p.win_Wp;

    if (warp == C::W_STRIP) {
        // ------------------------------------------------------------------ strip producer
        int it = 0;
        bool failed = false;
        const uint32_t strip_tx = (uint32_t)(p.win_srows * Wp * 128);
        for (int t = unit0; t < total_units; t += nunits) {
            const int m_tile = t * CG + rank;
            const int L0 = m_tile * p.win_tile;
            const int g0 = L0 / Wp;
            // rank 1: rows between its strip and rank 0's, so that both tiles sit at rank 0's offsets
            const int shift = (CG == 2 && rank == 1) ? ((L0 - p.win_tile) % Wp) - (L0 % Wp) : 0;
            for (int cb = 0; cb < CB; ++cb, ++it) {
                const int s = it & 1;
                const uint32_t ok = mbar_wait_warp(&sempty[s], ((it >> 1) & 1) ^ 1, &abort_flag);
                if (__any_sync(0xffffffffu, ok == 0u)) {
                    failed = true;
                    break;
                }
                uint8_t* dst = strip + s * strip_stride + shift * 128;
                uint32_t fb = smem_u32(&sfull[s]);
                if (CG == 1 || rank == 0) mbar_arrive_expect_tx_elect(&sfull[s], (uint32_t)CG * strip_tx);
                if (CG == 2) fb = mapa_shared(fb, 0);
                for (int r = 0; r < p.win_srows; ++r) {
                    const int g = g0 + r;
                    const int n = g / p.win_Hp, hp = g - n * p.win_Hp;
                    // padded row hp of image n = input row hp - ph from column -pw (padding rows and
                    // columns, and images past the batch, are outside the tensor and arrive as zeros)
                    tma_load_4d_cg<CG>(dst + r * Wp * 128, &tmA, fb, cb * 64, -p.win_pw, hp - p.win_ph, n);
                }
            }
            if (failed) break;
        }
        if (failed) {
            if (lane == 0) report_timeout(&abort_flag);
            if (CG == 1 || rank == 0) {
                for (int i = it - 1; i >= 0 && i >= it - 2; --i) (void)mbar_drain_warp(&sfull[i & 1], (i >> 1) & 1);
            } else {
                // rank 1's copies complete on rank 0's barriers: give them a fixed time instead
                const uint64_t t0 = globaltimer();
                while (globaltimer() - t0 < 1000000ull) {
                }
            }
        }
    } else if (warp == C::W_WEIGHT) {
        // ------------------------------------------------------------------ weight producer
        if (RES) {
            uint32_t fb = smem_u32(&bfull[0]);
            if (CG == 1 || rank == 0) mbar_arrive_expect_tx_elect(&bfull[0], (uint32_t)(CG * ntaps * CB * BT));
            if (CG == 2) fb = mapa_shared(fb, 0);
            for (int tap = 0; tap < ntaps; ++tap)
                for (int cb = 0; cb < CB; ++cb)
                    win_load_wtile<BN, DG, CG>(p, &tmB, sgen + (tap * CB + cb) * BT, fb, tap, cb, 0, rank);
            if (CG == 1 || rank == 0) (void)mbar_drain_warp(&bfull[0], 0);
        } else {
            int bt = 0;
            bool failed = false;
            for (int t = unit0; t < total_units && !failed; t += nunits)
                for (int cb = 0; cb < CB && !failed; ++cb)
                    for (int tap = 0; tap < ntaps; ++tap, ++bt) {
                        const int s = bt % kWinBStages;
                        const uint32_t ok =
                            mbar_wait_warp(&bempty[s], ((bt / kWinBStages) & 1) ^ 1, &abort_flag);
                        if (__any_sync(0xffffffffu, ok == 0u)) {
                            failed = true;
                            break;
                        }
                        uint32_t fb = smem_u32(&bfull[s]);
                        if (CG == 1 || rank == 0) mbar_arrive_expect_tx_elect(&bfull[s], (uint32_t)(CG * BT));
                        if (CG == 2) fb = mapa_shared(fb, 0);
                        win_load_wtile<BN, DG, CG>(p, &tmB, sgen + s * BT, fb, tap, cb, 0, rank);
                    }
            if (failed) {
                if (lane == 0) report_timeout(&abort_flag);
                if (CG == 1 || rank == 0) {
                    for (int i = bt - 1; i >= 0 && i >= bt - kWinBStages; --i)
                        (void)mbar_drain_warp(&bfull[i % kWinBStages], (i / kWinBStages) & 1);
                } else {
                    const uint64_t t0 = globaltimer();
                    while (globaltimer() - t0 < 1000000ull) {
                    }
                }
            }
        }
    } else if (warp == C::W_MMA) {
        // ------------------------------------------------------------------ MMA issuer (rank 0 of a pair)
        const uint32_t idesc = idesc_act(BM * CG, BN, 0u, DG ? 1u : 0u);
        int it = 0, bt = 0, lt = 0;
        bool failed = false;
        if (RES && (CG == 1 || rank == 0)) {
            const uint32_t ok = mbar_wait_warp(&bfull[0], 0, &abort_flag);
            failed = __any_sync(0xffffffffu, ok == 0u);
        }
        for (int t = unit0; t < total_units && (CG == 1 || rank == 0) && !failed; t += nunits, ++lt) {
            const int buf = lt % C::NB;
            const uint32_t ok = mbar_wait_warp(&acce_bar[buf], ((lt / C::NB) & 1) ^ 1, &abort_flag);
            if (__any_sync(0xffffffffu, ok == 0u)) {
                failed = true;
                break;
            }
            tc_fence_after();
            const int L0 = t * CG * p.win_tile;  // this CTA's (rank 0's) tile
            const int off0 = L0 - (L0 / Wp) * Wp;  // tile start within the strip's first row
            const uint32_t d = tmem + (uint32_t)(buf * kWinACC * BN);
            for (int cb = 0; cb < CB && !failed; ++cb, ++it) {
                const int s = it & 1;
                const uint32_t oks = mbar_wait_warp(&sfull[s], (it >> 1) & 1, &abort_flag);
                if (__any_sync(0xffffffffu, oks == 0u)) {
                    failed = true;
                    break;
                }
                tc_fence_after();
                const uint32_t sa = smem_u32(strip + s * strip_stride);
                int r = 0, sx = 0;  // (tap / S, tap % S), stepped without divisions
#pragma unroll 1
                for (int tap = 0; tap < ntaps; ++tap) {
                    uint32_t sb;
                    int bs = 0;
                    if (RES) {
                        sb = sbase + (uint32_t)((tap * CB + cb) * BT);
                    } else {
                        bs = bt % kWinBStages;
                        const uint32_t okb = mbar_wait_warp(&bfull[bs], (bt / kWinBStages) & 1, &abort_flag);
                        if (__any_sync(0xffffffffu, okb == 0u)) {
                            failed = true;
                            break;
                        }
                        tc_fence_after();
                        sb = sbase + (uint32_t)(bs * BT);
                    }
                    const uint32_t a0 = sa + (uint32_t)((off0 + r * Wp + sx) * 128);
                    // K-step j of accumulator a: A rows a*128.. of the shifted strip, 32 bytes per K-step;
                    // B K-major (32 bytes per K-step) or, for the data gradient, MN-major (2 KB per K-step)
                    static_assert(kWinACC == 2, "two accumulators per MMA group");
                    const uint64_t ad = smem_desc(a0, 16, 1024, kSwizzle128B);
                    const uint64_t bd = DG ? smem_desc(sb, 8192, 1024, kSwizzle128B) : smem_desc(sb, 16, 1024, kSwizzle128B);
                    mma_act_x8_elect_cg<CG>(d, d + BN, ad, (128 * 128) >> 4, 32 >> 4, bd, DG ? (2048 >> 4) : (32 >> 4),
                                             idesc, (cb > 0 || tap > 0) ? 1u : 0u);
                    if (!RES) {
                        mma_commit_elect_cg<CG>(&bempty[bs], kAll);
                        ++bt;
                    }
                    if (++sx == p.win_S) {
                        sx = 0;
                        ++r;
                    }
                }
                mma_commit_elect_cg<CG>(&sempty[s], kAll);
            }
            mma_commit_elect_cg<CG>(&accf_bar[buf], kAll);  // arrives when this unit's MMAs have completed
        }
        if (CG == 1 || rank == 0) {
            if (failed && lane == 0) report_timeout(&abort_flag);
            mma_commit_elect_cg<CG>(&drain_bar, 1);
            (void)mbar_drain_warp(&drain_bar, 0);
        }
    } else {
        // ------------------------------------------------------------------ epilogue (warps 0 .. EPI-1)
        constexpr int CW = C::CW;
        const int quarter = warp & 3, col0 = (warp >> 2) * CW;  // TMEM lanes 32*quarter.., columns col0..
        float* st_tile = epi_tile + warp * 32 * 33;
        float* wsum = epi_sum + warp * 2 * p.Ncols;
        RowStats<CW> rs;
        rs.zero();
        const int img = p.win_Hp * Wp;
        int lt = 0;
        for (int t = unit0; t < total_units; t += nunits, ++lt) {
            const int m_tile = t * CG + rank;
            const int buf = lt % C::NB;
            const uint32_t ok = mbar_wait_warp(&accf_bar[buf], (lt / C::NB) & 1, &abort_flag);
            if (__any_sync(0xffffffffu, ok == 0u)) {
                if (lane == 0) report_timeout(&abort_flag);
                break;
            }
            tc_fence_after();
            const int row = quarter * 32 + lane;
            bool valid[kWinACC];
            int64_t out_row[kWinACC];
#pragma unroll
            for (int a = 0; a < kWinACC; ++a) {
                const int L = m_tile * p.win_tile + a * 128 + row;
                const int n = L / img, rem = L - n * img;
                const int hp = rem / Wp, wp = rem - hp * Wp;
                // rows past the tile belong to the next tile (row-aligned tiles are shorter than 256)
                valid[a] = m_tile < p.total_tiles && a * 128 + row < p.win_tile && n < p.gN && hp < p.win_P &&
                           wp < p.win_Q;
                out_row[a] = ((int64_t)n * p.win_P + hp) * p.win_Q + wp;
            }
            // chunks c = (accumulator, 32 of this warp's columns)
            const uint32_t taddr = tmem + ((uint32_t)(quarter * 32) << 16) + (uint32_t)(buf * kWinACC * BN + col0);
            constexpr int NCH = CW / 32, NC = kWinACC * NCH;
            // the next chunk's TMEM load in flight while this one is converted and stored
            uint32_t va[32], vb[32];
            tmem_ld_32x32b_x32(taddr, va);
#pragma unroll
            for (int c = 0; c < NC; ++c) {
                uint32_t(&cur)[32] = (c & 1) ? vb : va;
                uint32_t(&nxt)[32] = (c & 1) ? va : vb;
                tmem_ld_wait_regs(cur);
                const int a = c / NCH, ch = c % NCH;
                if (c + 1 < NC)
                    tmem_ld_32x32b_x32(taddr + (uint32_t)(((c + 1) / NCH) * BN + ((c + 1) % NCH) * 32), nxt);
                float back[32];
                store_row_chunk_act(p, cur, valid[a], out_row[a], col0 + ch * 32, back);
                if (want_stats) rs.add(ch, back, lane);
            }
            tc_fence_before();
            __syncwarp();
            if (lane == 0) {
                if constexpr (CG == 2)
                    mbar_arrive_cluster(mapa_shared(smem_u32(&acce_bar[buf]), 0));
                else
                    mbar_arrive(&acce_bar[buf]);
            }
        }
        if (want_stats) {
            rs.flush(st_tile, wsum, p.Ncols, col0, lane);  // the window kernel has one column tile
            asm volatile("bar.sync 1, %0;" ::"r"(C::EPI * 32) : "memory");
            float* dst = p.stats + (int64_t)blockIdx.x * 2 * p.Ncols;
            const int nc = 2 * p.Ncols;
            // warps 4g..4g+3 hold column group g; the other groups' rows are zero
            for (int c = threadIdx.x; c < nc; c += C::EPI * 32) {
                float v = (epi_sum[c] + epi_sum[nc + c]) + (epi_sum[2 * nc + c] + epi_sum[3 * nc + c]);
                if constexpr (C::EPI == 8)
                    v += (epi_sum[4 * nc + c] + epi_sum[5 * nc + c]) + (epi_sum[6 * nc + c] + epi_sum[7 * nc + c]);
                dst[c] = v;
            }
        }
    }
    tc_fence_before();
    __syncthreads();
    // neither CTA of a pair leaves while the other may still signal its barriers or read its TMEM
    if constexpr (CG == 2) cluster_sync_all();
    if (warp == C::W_MMA) {
        tc_fence_after();
        tmem_dealloc_cg<CG>(tmem, C::TMEM_COLS);
    }
}

// ----------------------------------------------------------------------------- window weight gradient
// dW[k][r][s][c] = sum over positions L of dy[L][k] * x_pad[L + r*Wp + s][c] for stride-1
// layers with 64 input and 64 output channels and at most 10 taps, in the padded position space
// of conv_win_kernel: dy is zero at the positions that are not outputs (its strip rows are read
// with w from 0 to Wp-1 and h from 0 to Hp-1, and the zero fill of TMA covers w >= Q and h >= P).
// A CTA owns all taps*64 x 64 outputs, as ceil(taps/2) 128 x 64 TMEM accumulators (tap pairs
// (0,1), (2,3), ...), and one contiguous range of K-blocks (256 positions, or two whole padded
// rows when those are a multiple of 16; split-K over CTAs, fixed-order reduce afterwards).  Per
// K-block it loads one x strip and one dy strip; all taps read the same x strip.  A operand (x,
// MN-major: a 128-byte strip row holds the 64 channels of one position) of tap pair (t0, t1):
// start row off(t0) + 16j for K-step j, second 64-row half LBO = (off(t1) - off(t0)) rows
// further; for an odd tap count the last pair's second half is computed and not stored.
// B operand (dy, MN-major): start row 16j.
constexpr int kWgWinKB = 256;  // positions per K-block (row-aligned K-blocks may be shorter)

template <int NACC>  // accumulators: ceil(taps / 2)
__global__ void __launch_bounds__(kWinThreads, 1)
    conv_wgwin_kernel(const __grid_constant__ CUtensorMap tmX, const __grid_constant__ CUtensorMap tmDY,
                      const ConvParams p)
{
    dbl::dev::grid_dependency_trigger();  // a convolution launched next may start its set-up
    extern __shared__ uint8_t smem_raw[];
    __shared__ __align__(8) uint64_t full_bar[2], empty_bar[2], accf_bar, acce_bar, drain_bar;
    __shared__ uint32_t tmem_slot;
    __shared__ volatile int abort_flag;

    const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
    const uint32_t sbase = (smem_u32(smem_raw) + 1023u) & ~1023u;
    uint8_t* sgen = smem_raw + (sbase - smem_u32(smem_raw));
    const int Wp = p.win_Wp;
    const int xalign = ((p.win_srows * Wp * 128 + 1023) / 1024) * 1024;  // dy strip offset in a stage
    const int stage_bytes = p.win_strip_bytes;
    const int ntaps = p.win_R * p.win_S;

    if (threadIdx.x == 0) {
        for (int i = 0; i < 2; ++i) {
            mbar_init(&full_bar[i], 2);  // one expect_tx arrival per producer warp
            mbar_init(&empty_bar[i], 1);
        }
        mbar_init(&accf_bar, 1);
        mbar_init(&acce_bar, 4);
        mbar_init(&drain_bar, 1);
        abort_flag = 0;
        fence_mbar_init();
    }
    if ((warp == 4 || warp == 5) && lane == 0) tma_prefetch_desc(warp == 4 ? &tmX : &tmDY);
    if (warp == 6) {
        tmem_alloc(&tmem_slot, 512);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    grid_dependency_wait();  // the set-up above may overlap the previous kernel; memory only after it
    const uint32_t tmem = tmem_slot;

    if (warp == 4 || warp == 5) {
        // ------------------------------------------------------------------ producers: x rows (4), dy rows (5)
        const bool is_x = warp == 4;
        const int rows = is_x ? p.win_srows : p.win_dyrows;
        const uint32_t tx = (uint32_t)(rows * Wp * 128);
        int it = 0;
        bool failed = false;
        for (int z = blockIdx.x; z < p.zdim && !failed; z += gridDim.x) {
            const int kb0 = z * p.kb_per_split, kb1 = min(p.num_kb, kb0 + p.kb_per_split);
            for (int kb = kb0; kb < kb1; ++kb, ++it) {
                const int s = it & 1;
                const uint32_t ok = mbar_wait_warp(&empty_bar[s], ((it >> 1) & 1) ^ 1, &abort_flag);
                if (__any_sync(0xffffffffu, ok == 0u)) {
                    failed = true;
                    break;
                }
                uint8_t* dst = sgen + s * stage_bytes + (is_x ? 0 : xalign);
                const int g0 = kb * p.win_tile / Wp;
                mbar_arrive_expect_tx_elect(&full_bar[s], tx);
                for (int r = 0; r < rows; ++r) {
                    const int g = g0 + r;
                    const int n = g / p.win_Hp, hp = g - n * p.win_Hp;
                    if (is_x)
                        tma_load_4d_elect(dst + r * Wp * 128, &tmX, &full_bar[s], 0, -p.win_pw, hp - p.win_ph, n);
                    else
                        tma_load_4d_elect(dst + r * Wp * 128, &tmDY, &full_bar[s], 0, 0, hp, n);
                }
            }
        }
        if (failed) {
            if (lane == 0) report_timeout(&abort_flag);
            for (int i = it - 1; i >= 0 && i >= it - 2; --i) (void)mbar_drain_warp(&full_bar[i & 1], (i >> 1) & 1);
        }
    } else if (warp == 6) {
        // ------------------------------------------------------------------ MMA issuer
        const uint32_t idesc = idesc_act(BM, 64, 1u, 1u);
        // strip-row offsets of each tap pair's two halves (the unused half of an odd last pair
        // reads the row after its first half), once per CTA
        int o0[NACC], o1[NACC];
#pragma unroll
        for (int pp = 0; pp < NACC; ++pp) {
            const int t0 = 2 * pp, t1 = 2 * pp + 1;
            o0[pp] = (t0 / p.win_S) * Wp + t0 % p.win_S;
            o1[pp] = t1 < ntaps ? (t1 / p.win_S) * Wp + t1 % p.win_S : o0[pp] + 1;
        }
        int it = 0, lt = 0;
        bool failed = false;
        for (int z = blockIdx.x; z < p.zdim && !failed; z += gridDim.x, ++lt) {
            const uint32_t ok = mbar_wait_warp(&acce_bar, (lt & 1) ^ 1, &abort_flag);
            if (__any_sync(0xffffffffu, ok == 0u)) {
                failed = true;
                break;
            }
            tc_fence_after();
            const int kb0 = z * p.kb_per_split, kb1 = min(p.num_kb, kb0 + p.kb_per_split);
            for (int kb = kb0; kb < kb1; ++kb, ++it) {
                const int s = it & 1;
                const uint32_t okf = mbar_wait_warp(&full_bar[s], (it >> 1) & 1, &abort_flag);
                if (__any_sync(0xffffffffu, okf == 0u)) {
                    failed = true;
                    break;
                }
                tc_fence_after();
                const int P0 = kb * p.win_tile;
                const int off = P0 - (P0 / Wp) * Wp;
                const uint32_t xa = sbase + (uint32_t)(s * stage_bytes), ya = xa + (uint32_t)xalign;
#pragma unroll 1
                for (int j = 0; j < p.win_tile / 16; ++j) {
                    const uint64_t bd = smem_desc(ya + (uint32_t)((off + 16 * j) * 128), 16384, 1024, kSwizzle128B);
#pragma unroll
                    for (int pp = 0; pp < NACC; ++pp) {
                        const uint64_t ad = smem_desc(xa + (uint32_t)((off + o0[pp] + 16 * j) * 128),
                                                      (uint32_t)((o1[pp] - o0[pp]) * 128), 1024, kSwizzle128B);
                        mma_act_elect(tmem + (uint32_t)(pp * 64), ad, bd, idesc, (kb > kb0 || j > 0) ? 1u : 0u);
                    }
                }
                mma_commit_elect(&empty_bar[s]);
            }
            mma_commit_elect(&accf_bar);  // arrives when this split's MMAs have completed
        }
        if (failed && lane == 0) report_timeout(&abort_flag);
        mma_commit_elect(&drain_bar);
        (void)mbar_drain_warp(&drain_bar, 0);
    } else {
        // ------------------------------------------------------------------ epilogue (warps 0-3)
        const int i = warp * 32 + lane;  // TMEM lane = accumulator row
        int lt = 0;
        for (int z = blockIdx.x; z < p.zdim; z += gridDim.x, ++lt) {
            const uint32_t ok = mbar_wait_warp(&accf_bar, lt & 1, &abort_flag);
            if (__any_sync(0xffffffffu, ok == 0u)) {
                if (lane == 0) report_timeout(&abort_flag);
                break;
            }
            tc_fence_after();
            const int kb0 = z * p.kb_per_split;
            const bool have_acc = min(p.num_kb, kb0 + p.kb_per_split) > kb0;
#pragma unroll 1
            for (int pp = 0; pp < NACC; ++pp) {
                const int tap = 2 * pp + (i >> 6), c = i & 63;
                const bool valid = tap < ntaps;
                const int m = tap * 64 + c;  // row of dW viewed as [k][(r, s, c)]
#pragma unroll 1
                for (int ch = 0; ch < 2; ++ch) {
                    uint32_t v[32];
                    if (have_acc) {
                        tmem_ld_32x32b_x32(tmem + ((uint32_t)(warp * 32) << 16) + (uint32_t)(pp * 64 + ch * 32), v);
                        tmem_ld_wait();
                    } else {
#pragma unroll
                        for (int k = 0; k < 32; ++k) v[k] = 0u;
                    }
                    if (valid) {
                        // [slice][k][m]: consecutive lanes hold consecutive m, one 128-byte line per store
                        float* o = static_cast<float*>(p.out) + ((int64_t)(p.zdim > 1 ? z : 0) * 64 + ch * 32) * p.M + m;
                        if (p.zdim == 1 && p.wg_accumulate) {
#pragma unroll
                            for (int k = 0; k < 32; ++k) o[(int64_t)k * p.M] += __uint_as_float(v[k]);
                        } else {
#pragma unroll
                            for (int k = 0; k < 32; ++k) o[(int64_t)k * p.M] = __uint_as_float(v[k]);
                        }
                    }
                }
            }
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(&acce_bar);
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 6) {
        tc_fence_after();
        tmem_dealloc(tmem, 512);
    }
}

// ----------------------------------------------------------------------------- reductions
// Per-output-channel sums of the conv epilogue's per-CTA partials part[nparts][2][K]
// (partials_colsum, fixed order).
__global__ void __launch_bounds__(kPartialsThreads) stats_reduce_kernel(const float* __restrict__ part, int nparts, int K,
                                                           float* __restrict__ sum, float* __restrict__ sumsq)
{
    double s, q;
    const int c = partials_colsum(part, nparts, K, s, q);
    if (c >= 0) {
        sum[c] = (float)s;
        sumsq[c] = (float)q;
    }
}

// dw[i] (+)= sum over slices of part[slice][i] in a fixed order; i runs over
// the KRSC weight gradient (the slices are already in that layout).  LANES
// threads share one float4 of dw: thread j sums slices j, j+LANES, ... (four
// loads in flight), then a fixed shuffle tree adds the LANES partial sums.
// LANES = 1 for a few slices, 8 for many (the 64-channel layers split K ~60 ways).
template <int LANES>
__global__ void __launch_bounds__(256) wgrad_reduce_kernel(const float* __restrict__ part, int slices, int64_t n,
                                                           float* __restrict__ dw, int accumulate)
{
    dbl::dev::grid_dependency_trigger();  // a convolution launched next may start its set-up
    const int j = threadIdx.x % LANES;
    const int64_t n4 = n >> 2;
    const int64_t groups = blockDim.x / LANES;
    // the loop bound is the same for the whole block, so every shuffle sees all 32 lanes
    for (int64_t base = (int64_t)blockIdx.x * groups; base < n4; base += (int64_t)gridDim.x * groups) {
        const int64_t i = base + threadIdx.x / LANES;
        const int sl = i < n4 ? slices : 0;  // groups past the end add nothing and store nothing
        float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
        int s = j;
        for (; s + 3 * LANES < sl; s += 4 * LANES) {
            float4 v[4];
#pragma unroll
            for (int u = 0; u < 4; ++u)
                v[u] = __ldcs(reinterpret_cast<const float4*>(part + (int64_t)(s + u * LANES) * n) + i);
#pragma unroll
            for (int u = 0; u < 4; ++u) {
                acc.x += v[u].x;
                acc.y += v[u].y;
                acc.z += v[u].z;
                acc.w += v[u].w;
            }
        }
        for (; s < sl; s += LANES) {
            const float4 v = __ldcs(reinterpret_cast<const float4*>(part + (int64_t)s * n) + i);
            acc.x += v.x;
            acc.y += v.y;
            acc.z += v.z;
            acc.w += v.w;
        }
#pragma unroll
        for (int o = LANES / 2; o; o >>= 1) {
            acc.x += __shfl_xor_sync(0xffffffffu, acc.x, o, LANES);
            acc.y += __shfl_xor_sync(0xffffffffu, acc.y, o, LANES);
            acc.z += __shfl_xor_sync(0xffffffffu, acc.z, o, LANES);
            acc.w += __shfl_xor_sync(0xffffffffu, acc.w, o, LANES);
        }
        if (j == 0 && i < n4) {
            float4* d = reinterpret_cast<float4*>(dw) + i;
            if (accumulate) {
                const float4 o = *d;
                acc.x += o.x;
                acc.y += o.y;
                acc.z += o.z;
                acc.w += o.w;
            }
            *d = acc;
        }
    }
    const int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    for (int64_t i = (n4 << 2) + t; i < n; i += (int64_t)gridDim.x * blockDim.x) {
        float acc = 0.f;
        for (int s = 0; s < slices; ++s) acc += part[(int64_t)s * n + i];
        dw[i] = accumulate ? dw[i] + acc : acc;
    }
}

// ----------------------------------------------------------------------------- host side
struct Plan {
    int mode;
    int BN;
    int cg = 1;          // conv_igemm_kernel CTAs per tile (2: CTA pairs with M = 256 MMAs)
    ConvParams p;
    size_t ws_main = 0;  // bytes: fwd channel-sum partials, or wgrad split-K slices
    bool win = false;    // conv_win_kernel (3x3 stride-1 correlation over padded strips)
    bool res = false;    // window kernel with all weights resident in shared memory
    size_t smem = 0;     // window kernel dynamic shared memory
};



int out_dim(int in, int k, int st, int pad) { return (in + 2 * pad - k) / st + 1; }

int fwd_tile_rows(int BN);

int choose_bn(int cols)
{
    if (cols % 256 == 0) return 256;
    if (cols % 128 == 0) return 128;
    return 64;
}

// Strides and pads per axis (stride_w == 0 means: the same as along H).
struct Geom {
    int sh, sw, ph, pw;
};

Geom geom(const dbl_conv_shape* s)
{
    Geom g{s->stride, s->stride_w ? s->stride_w : s->stride, s->pad, s->stride_w ? s->pad_w : s->pad};
    return g;
}

int validate(const dbl_conv_shape* s, const char* who)
{
    using dbl::set_error;
    if (!s) return set_error(DBL_ERR_INVALID, "%s: null shape", who);
    const Geom g = geom(s);
    if (s->n <= 0 || s->h <= 0 || s->w <= 0 || s->c <= 0 || s->k <= 0 || s->r <= 0 || s->s <= 0 || g.sh <= 0 ||
        g.sw <= 0 || g.ph < 0 || g.pw < 0)
        return set_error(DBL_ERR_INVALID, "%s: non-positive dimension", who);
    if (s->c % 8) return set_error(DBL_ERR_INVALID, "%s: channels must be a multiple of 8", who);
    if (s->k % 64) return set_error(DBL_ERR_UNSUPPORTED, "%s: output channels must be a multiple of 64", who);
    if (s->k > kMaxNcols || s->c > kMaxNcols * 8)
        return set_error(DBL_ERR_UNSUPPORTED, "%s: at most %d output channels", who, kMaxNcols);
    if (g.sh > 2 || g.sw > 2 || s->r > 8 || s->s > 8 || g.ph > 3 || g.pw > 3)
        return set_error(DBL_ERR_UNSUPPORTED, "%s: stride <= 2, filter <= 8, pad <= 3 per axis supported", who);
    if (out_dim(s->h, s->r, g.sh, g.ph) <= 0 || out_dim(s->w, s->s, g.sw, g.pw) <= 0)
        return set_error(DBL_ERR_INVALID, "%s: empty output", who);
    return DBL_OK;
}

// Split-K slices of the implicit-GEMM weight gradient: the count that minimises the
// modelled time of the persistent grid on a 152-SM GPU, where the busiest CTA runs
// ceil(units / 152) units of (K-blocks per slice + ~2 K-blocks of epilogue) and the
// fixed-order reduce afterwards reads every slice (one K-block of a 128 x BN tile is
// ~4 BN tensor cycles, in which the GPU streams ~10.5 KB x BN).  At least 4 K-blocks
// (512 pixels) per slice.  A fixed function of the shape, so the summation order, and
// with it the result, does not depend on the device the plan runs on.
int wgrad_splits(int tiles, int num_kb, int rows, int cols, int BN, int cg)
{
    const int kPlanSMs = 152 / cg;  // tile processors: SMs, or SM pairs
    const double slice_cost = (double)rows * cols * 4 / (10.5e3 * BN);  // K-block times to reduce one slice
    int best = 1;
    double best_cost = 1e300;
    const int max_splits = std::max(1, num_kb / 4);
    for (int sp = 1; sp <= max_splits; ++sp) {
        const int kbs = (num_kb + sp - 1) / sp;
        const int eff = (num_kb + kbs - 1) / kbs;  // slices actually used
        if (eff != sp) continue;
        const int rounds = (tiles * sp + kPlanSMs - 1) / kPlanSMs;
        const double cost = rounds * (kbs + 2.0) + (sp > 1 ? sp * slice_cost : 0.0);
        if (cost < best_cost) {
            best_cost = cost;
            best = sp;
        }
    }
    return best;
}

// Persistent grid: one CTA per SM (the kernel uses ~225 KB of shared memory), never more
// CTAs than tiles, never more than kMaxGrid (the workspace is sized for that bound).
int grid_size(int total_tiles)
{
    int g = dbl::sm_count();
    if (g > kMaxGrid) g = kMaxGrid;
    if (g > total_tiles) g = total_tiles;
    return g < 1 ? 1 : g;
}

// Dynamic shared memory the window kernel may use (227 KB per CTA, less the
// static barriers and 1 KB of alignment slack).
constexpr size_t kWinSmemMax = 232448 - 2048;

// Positions per tile of the window kernels: 256 (any start), or, for rows of at
// least 64 positions, the whole rows that fit in 256 (row-aligned starts need no
// strip row for a misaligned start).
int win_tile_positions(int Wp) { return Wp >= 64 ? (kWinBMT / Wp) * Wp : kWinBMT; }

// Window-kernel eligibility and geometry (see conv_win_kernel): stride 1 on both
// axes, 64-channel blocks of the reduced operand (red_c), 64 or 128 output
// channels, padded rows of 10..256 positions; the data gradient (dgrad) for
// 3x3 filters with pad 1 only (its taps are the forward taps flipped).
bool win_pairs();
int cta_pair_level();

bool win_setup(const dbl_conv_shape* s, int red_c, int out_c, bool dgrad, Plan& pl)
{
    const Geom g = geom(s);
    if (g.sh != 1 || g.sw != 1) return false;
    if (dgrad && (s->r != 3 || s->s != 3 || g.ph != 1 || g.pw != 1)) return false;
    if (s->r * s->s > 16 || red_c % 64 != 0 || (out_c != 64 && out_c != 128)) return false;
    const int Wp = s->w + 2 * g.pw, Hp = s->h + 2 * g.ph;
    if (Wp < 10 || Wp > 256) return false;
    const int P = Hp - s->r + 1, Q = Wp - s->s + 1;
    if (P <= 0 || Q <= 0) return false;
    const int64_t L = (int64_t)s->n * Hp * Wp;
    if (L > INT32_MAX / 4) return false;
    const int tile = win_tile_positions(Wp);
    // rows one tile's 256 accumulator rows read: start offset within a row, plus 255, plus the last tap's offset
    const int max_index = (tile % Wp == 0 ? 0 : Wp - 1) + kWinBMT - 1 + (s->r - 1) * Wp + (s->s - 1);
    const int srows = max_index / Wp + 1;
    const int strip = ((srows * Wp * 128 + 1023) / 1024) * 1024;
    const int BN = out_c, CB = red_c / 64, ntaps = s->r * s->s;
    const bool res = BN == 64 && CB == 1 && ntaps <= 9;
    // CTA pairs for 128-column tiles: each SM stages half of the weights; rank 1's strip is
    // shifted by up to a padded row either way, so each strip buffer gets a margin of one padded
    // row on both sides (single CTAs when the pair layout does not fit in shared memory).  The
    // 64-column forward pass with resident weights runs on pairs only with DBL_CONV_CTA_PAIRS=2:
    // it halves each SM's weight reads (a sixth of its tensor-core shared-memory reads) but
    // couples the two CTAs' loads and epilogues; with two accumulator buffers it measured slower
    // (layer1 forward at batch 384: 113 against 97 us), with four the same (122 against 123 us
    // at batch 512).
    if ((size_t)srows * Wp * 128 >= (1u << 20)) return false;
    const int epi = out_c == 64 ? WinCfg<64>::EPI : WinCfg<128>::EPI;
    int cg = win_pairs() && (BN == 128 || (BN == 64 && res && !dgrad && cta_pair_level() == 2)) ? 2 : 1;
    int margin = 0;
    size_t smem = 0;
    for (;; cg = 1) {
        margin = cg == 2 ? (Wp * 128 + 1023) / 1024 * 1024 : 0;
        const int b_bytes = (res ? ntaps * CB * WinCfg<64>::B_TILE : kWinBStages * BN * 128) / cg;
        // epilogue statistics: per-warp channel sums after the strips (the warps' transposes reuse the strips)
        const size_t strips = 2 * ((size_t)strip + 2 * (size_t)margin);
        smem = (size_t)b_bytes + strips + (size_t)epi * 2 * out_c * 4 + 1024;
        if (strips >= (size_t)epi * 32 * 33 * 4 && smem <= kWinSmemMax) break;
        if (cg == 1) return false;
    }
    ConvParams& p = pl.p;
    pl.win = true;
    pl.res = res;
    pl.BN = BN;
    pl.cg = cg;
    pl.smem = smem;
    p.win_margin = margin;
    p.win_R = s->r;
    p.win_S = s->s;
    p.win_ph = g.ph;
    p.win_pw = g.pw;
    p.win_P = P;
    p.win_Q = Q;
    p.win_Hp = Hp;
    p.win_Wp = Wp;
    p.win_tile = tile;
    p.win_srows = srows;
    p.win_strip_bytes = strip;
    p.M = s->n * P * Q;
    p.m_tiles = (int)((L + tile - 1) / tile);
    p.n_tiles = 1;
    p.cblocks = CB;
    p.gN = s->n;
    p.Ncols = out_c;
    p.ldo = out_c;
    p.Cin = red_c;
    return true;
}

// Window weight-gradient eligibility and geometry (see conv_wgwin_kernel):
// stride 1, 64 input and 64 output channels, at most 10 taps, padded rows of
// 10..256 positions.
bool wgwin_setup(const dbl_conv_shape* s, Plan& pl)
{
    const Geom g = geom(s);
    if (g.sh != 1 || g.sw != 1) return false;
    if (s->c != 64 || s->k != 64) return false;
    const int ntaps = s->r * s->s;
    if ((ntaps + 1) / 2 != 2 && (ntaps + 1) / 2 != 5) return false;  // the instantiated accumulator counts
    const int Wp = s->w + 2 * g.pw, Hp = s->h + 2 * g.ph;
    if (Wp < 10 || Wp > 256) return false;
    const int P = Hp - s->r + 1, Q = Wp - s->s + 1;
    if (P <= 0 || Q <= 0) return false;
    const int64_t L = (int64_t)s->n * Hp * Wp;
    if (L > INT32_MAX / 4) return false;
    // K-block: two whole padded rows when that is a multiple of 16 positions (no misaligned start), else 256
    const int kb = (Wp >= 64 && 2 * Wp <= kWgWinKB && (2 * Wp) % 16 == 0) ? 2 * Wp : kWgWinKB;
    const int start = kb % Wp == 0 ? 0 : Wp - 1;
    auto off = [&](int t) { return (t / s->s) * Wp + t % s->s; };
    const int last = (ntaps % 2) ? off(ntaps - 1) + 1 : off(ntaps - 1);  // the unused half of an odd last pair
    const int xrows = (start + kb - 1 + last) / Wp + 1;
    const int dyrows = (start + kb - 1) / Wp + 1;
    const int xalign = ((xrows * Wp * 128 + 1023) / 1024) * 1024;
    const int stage = xalign + ((dyrows * Wp * 128 + 1023) / 1024) * 1024;
    const size_t smem = 2 * (size_t)stage + 1024;
    if (smem > kWinSmemMax) return false;
    ConvParams& p = pl.p;
    pl.win = true;
    pl.BN = 64;
    pl.smem = smem;
    pl.mode = p.mode = kWgrad;
    p.win_R = s->r;
    p.win_S = s->s;
    p.win_ph = g.ph;
    p.win_pw = g.pw;
    p.win_P = P;
    p.win_Q = Q;
    p.win_Hp = Hp;
    p.win_Wp = Wp;
    p.win_tile = kb;
    p.win_srows = xrows;
    p.win_dyrows = dyrows;
    p.win_strip_bytes = stage;
    p.M = ntaps * 64;
    p.Ncols = 64;
    p.m_tiles = p.n_tiles = 1;
    p.gN = s->n;
    p.num_kb = (int)((L + kb - 1) / kb);
    // one contiguous range of K-blocks per CTA of a persistent grid
    int splits = grid_size(p.num_kb);
    p.kb_per_split = (p.num_kb + splits - 1) / splits;
    p.zdim = (p.num_kb + p.kb_per_split - 1) / p.kb_per_split;
    pl.ws_main = p.zdim > 1 ? (size_t)p.zdim * p.M * 64 * sizeof(float) : 0;
    return true;
}

// Which tiles run on CTA pairs (see conv_igemm_kernel): 256-column tiles, and the
// 128-column tiles of the weight gradient (its long K-blocks amortise the pair's
// extra synchronisation; the short-K forward and data-gradient passes of 128
// columns measured slower on pairs).  The environment variable DBL_CONV_CTA_PAIRS
// overrides this: 0 = never, 2 = every 128- and 256-column tile.
int cta_pair_level()
{
    static const int level = [] {
        const char* e = getenv("DBL_CONV_CTA_PAIRS");
        return e && (e[0] == '0' || e[0] == '2') ? e[0] - '0' : 1;
    }();
    return level;
}

bool pair_tiles(int BN, bool wgrad)
{
    const int level = cta_pair_level();
    if (level == 0) return false;
    return BN == 256 || (BN == 128 && (wgrad || level == 2));
}

// Window-kernel CTA pairs: 128-column tiles; with DBL_CONV_CTA_PAIRS=2 also the 64-column
// forward pass with resident weights (measured no faster, for comparison); DBL_CONV_CTA_PAIRS=0
// turns them off with the others.
bool win_pairs() { return cta_pair_level() != 0; }

int make_plan(const dbl_conv_shape* s, int pass, Plan& pl)
{
    using dbl::set_error;
    int rc = validate(s, pass == DBL_PASS_FWD ? "conv_fwd" : pass == DBL_PASS_DGRAD ? "conv_dgrad" : "conv_wgrad");
    if (rc) return rc;
    const Geom g = geom(s);
    const int P = out_dim(s->h, s->r, g.sh, g.ph), Q = out_dim(s->w, s->s, g.sw, g.pw);
    ConvParams& p = pl.p;
    memset(&p, 0, sizeof(p));
    const bool c8 = s->c == 8;
    if (!c8 && s->c % 64) return set_error(DBL_ERR_UNSUPPORTED, "conv: input channels must be 8 or a multiple of 64");
    p.ntaps = s->r * s->s;
    p.S = s->s;
    p.Cin = s->c;
    p.zdim = 1;
    if (pass == DBL_PASS_FWD && !c8 && win_setup(s, s->c, s->k, false, pl)) {
        pl.mode = p.mode = kFwd;
        pl.ws_main = (size_t)kMaxGrid * 2 * s->k * sizeof(float);
    } else if (pass == DBL_PASS_DGRAD && s->c % 64 == 0 && win_setup(s, s->k, s->c, true, pl)) {
        pl.mode = p.mode = kDgrad;
    } else if (pass == DBL_PASS_WGRAD && wgwin_setup(s, pl)) {
        // conv_wgwin_kernel: tiles are the split-K ranges
    } else if (pass == DBL_PASS_FWD) {
        pl.mode = p.mode = c8 ? kFwdC8 : kFwd;
        if (c8 && p.ntaps > 56) return set_error(DBL_ERR_UNSUPPORTED, "conv_fwd: stem filter too large");
        const int64_t M = (int64_t)s->n * P * Q;
        if (M > INT32_MAX / 2) return set_error(DBL_ERR_UNSUPPORTED, "conv_fwd: too many output pixels");
        p.M = (int)M;
        p.Ncols = s->k;
        pl.BN = c8 ? 64 : choose_bn(s->k);
        pl.cg = !c8 && pair_tiles(pl.BN, false) ? 2 : 1;
        p.m_tiles = (p.M + pl.cg * fwd_tile_rows(pl.BN) - 1) / (pl.cg * fwd_tile_rows(pl.BN));
        p.n_tiles = s->k / pl.BN;
        p.gN = s->n;
        p.gP = P;
        p.gQ = Q;
        p.tstride_h = g.sh;
        p.tstride_w = g.sw;
        p.base_h = -g.ph;
        p.base_w = -g.pw;
        p.cblocks = c8 ? 1 : s->c / 64;
        p.num_kb = c8 ? (p.ntaps + 7) / 8 : p.ntaps * p.cblocks;
        p.ldo = s->k;
        pl.ws_main = (size_t)kMaxGrid * 2 * s->k * sizeof(float);
    } else if (pass == DBL_PASS_DGRAD) {
        if (c8) return set_error(DBL_ERR_UNSUPPORTED, "conv_dgrad: the 8-channel stem has no data gradient path");
        if (s->r != s->s || g.sh != g.sw || g.ph != g.pw)
            return set_error(DBL_ERR_UNSUPPORTED, "conv_dgrad: square filters with equal strides and pads only");
        pl.mode = p.mode = kDgrad;
        p.Ncols = s->c;
        pl.BN = choose_bn(s->c);
        p.n_tiles = s->c / pl.BN;
        p.cblocks = s->k / 64;
        p.ldo = s->c;
        p.out_h = s->h;
        p.out_w = s->w;
        p.gN = s->n;
        if (s->stride == 1) {
            if (P != s->h || Q != s->w)
                return set_error(DBL_ERR_UNSUPPORTED, "conv_dgrad: stride 1 needs 'same' padding (P == H)");
            p.phase_div = 1;
            p.M = s->n * s->h * s->w;
            p.gP = s->h;
            p.gQ = s->w;
            p.base_h = p.base_w = -(s->r - 1 - s->pad);
            int t = 0;
            p.phase_off[0] = 0;
            for (int r2 = 0; r2 < s->r; ++r2)
                for (int s2 = 0; s2 < s->s; ++s2) {
                    if (t >= 16) return set_error(DBL_ERR_UNSUPPORTED, "conv_dgrad: too many taps");
                    // im2col offset (r2, s2) reads dy at h - (R-1-pad) + r2 = h + pad - r with r = R-1-r2
                    p.tap_oh[t] = (int8_t)r2;
                    p.tap_ow[t] = (int8_t)s2;
                    p.tap_r[t] = (int8_t)(s->r - 1 - r2);
                    p.tap_s[t] = (int8_t)(s->s - 1 - s2);
                    ++t;
                }
            p.phase_off[1] = t;
        } else {
            if ((s->h & 1) || (s->w & 1) || P * 2 != s->h || Q * 2 != s->w)
                return set_error(DBL_ERR_UNSUPPORTED, "conv_dgrad: stride 2 needs even H, W with P = H/2");
            for (int r = 0; r < s->r; ++r)
                if (r > 1 + s->pad) return set_error(DBL_ERR_UNSUPPORTED, "conv_dgrad: stride-2 filter too large for pad");
            p.phase_div = 2;
            p.zdim = 4;
            p.gP = s->h / 2;
            p.gQ = s->w / 2;
            p.M = s->n * p.gP * p.gQ;
            p.base_h = p.base_w = 0;
            int t = 0;
            for (int ph = 0; ph < 4; ++ph) {
                const int a = ph >> 1, b = ph & 1;
                p.phase_off[ph] = t;
                for (int r = 0; r < s->r; ++r) {
                    const int dh = a + s->pad - r;
                    if (dh < 0 || (dh & 1)) continue;
                    for (int c2 = 0; c2 < s->s; ++c2) {
                        const int dw = b + s->pad - c2;
                        if (dw < 0 || (dw & 1)) continue;
                        if (t >= 16) return set_error(DBL_ERR_UNSUPPORTED, "conv_dgrad: too many taps");
                        p.tap_r[t] = (int8_t)r;
                        p.tap_s[t] = (int8_t)c2;
                        p.tap_oh[t] = (int8_t)(dh / 2);
                        p.tap_ow[t] = (int8_t)(dw / 2);
                        ++t;
                    }
                }
            }
            p.phase_off[4] = t;
        }
        pl.cg = pair_tiles(pl.BN, false) ? 2 : 1;
        p.m_tiles = (p.M + pl.cg * fwd_tile_rows(pl.BN) - 1) / (pl.cg * fwd_tile_rows(pl.BN));
    } else {
        pl.mode = p.mode = c8 ? kWgradC8 : kWgrad;
        p.M = p.ntaps * s->c;  // D rows = (tap, c)
        p.Ncols = s->k;
        pl.BN = c8 ? 64 : choose_bn(s->k);
        pl.cg = !c8 && pair_tiles(pl.BN, true) ? 2 : 1;
        p.m_tiles = c8 ? (p.ntaps + 15) / 16 : (p.M + pl.cg * BM - 1) / (pl.cg * BM);
        p.n_tiles = s->k / pl.BN;
        p.gN = s->n;
        p.gP = P;
        p.gQ = Q;
        p.tstride_h = g.sh;
        p.tstride_w = g.sw;
        p.base_h = -g.ph;
        p.base_w = -g.pw;
        const int64_t pix = (int64_t)s->n * P * Q;
        if ((pix + 127) / 128 > INT32_MAX / 2) return set_error(DBL_ERR_UNSUPPORTED, "conv_wgrad: too many pixels");
        p.num_kb = (int)((pix + 127) / 128);  // K-blocks of 128 output pixels
        const int splits = wgrad_splits(p.m_tiles * p.n_tiles, p.num_kb, p.M, s->k, pl.BN, pl.cg);
        p.kb_per_split = (p.num_kb + splits - 1) / splits;
        p.zdim = splits;
        pl.ws_main = splits > 1 ? (size_t)splits * p.M * s->k * sizeof(float) : 0;
    }
    p.total_tiles = p.m_tiles * p.n_tiles * p.zdim;
    return DBL_OK;
}

size_t plan_ws(const Plan& pl) { return ((pl.ws_main + 255) / 256) * 256; }

// im2col tensor map over an NHWC tensor.  Bounding-box corners and traversal
// strides are given per spatial axis; the driver takes them innermost axis
// first (W, then H), like the tensor dimensions.
int enc_im2col(CUtensorMap* m, const void* base, int N, int H, int W, int C, int lower_h, int upper_h, int lower_w,
               int upper_w, int stride_h, int stride_w, int channels, int pixels, bool swizzle)
{
    auto fn = dbl::encode_im2col();
    if (!fn) return dbl::set_error(DBL_ERR_CUDA, "conv: cuTensorMapEncodeIm2col unavailable from the driver");
    cuuint64_t dims[4] = {(cuuint64_t)C, (cuuint64_t)W, (cuuint64_t)H, (cuuint64_t)N};
    cuuint64_t strides[3] = {(cuuint64_t)C * 2, (cuuint64_t)W * C * 2, (cuuint64_t)H * W * C * 2};
    int lo[2] = {lower_w, lower_h}, hi[2] = {upper_w, upper_h};
    cuuint32_t es[4] = {1, (cuuint32_t)stride_w, (cuuint32_t)stride_h, 1};
    CUresult r = fn(m, (dbl::act::kF16 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT16 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16), 4, const_cast<void*>(base), dims, strides, lo, hi,
                    (cuuint32_t)channels, (cuuint32_t)pixels, es, CU_TENSOR_MAP_INTERLEAVE_NONE,
                    swizzle ? CU_TENSOR_MAP_SWIZZLE_128B : CU_TENSOR_MAP_SWIZZLE_NONE,
                    CU_TENSOR_MAP_L2_PROMOTION_L2_128B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) return dbl::set_error(DBL_ERR_CUDA, "conv: im2col tensor map encode failed (%d)", (int)r);
    return DBL_OK;
}

int enc_tiled(CUtensorMap* m, const void* base, int rank, const cuuint64_t* dims, const cuuint64_t* strides_bytes,
              const cuuint32_t* box, bool swizzle)
{
    auto fn = dbl::encode_tiled();
    if (!fn) return dbl::set_error(DBL_ERR_CUDA, "conv: cuTensorMapEncodeTiled unavailable from the driver");
    cuuint32_t es[5] = {1, 1, 1, 1, 1};
    CUresult r = fn(m, (dbl::act::kF16 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT16 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16), (cuuint32_t)rank, const_cast<void*>(base), dims,
                    strides_bytes, box, es, CU_TENSOR_MAP_INTERLEAVE_NONE,
                    swizzle ? CU_TENSOR_MAP_SWIZZLE_128B : CU_TENSOR_MAP_SWIZZLE_NONE,
                    CU_TENSOR_MAP_L2_PROMOTION_L2_128B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) return dbl::set_error(DBL_ERR_CUDA, "conv: tiled tensor map encode failed (%d)", (int)r);
    return DBL_OK;
}

template <int BN, int FAM, int CG>
int set_igemm_smem()
{
    static bool attr_set[64] = {false};
    int dev = 0;
    cudaGetDevice(&dev);
    if (dev >= 0 && dev < 64 && !attr_set[dev]) {
        cudaError_t e = cudaFuncSetAttribute(conv_igemm_kernel<BN, FAM, CG>,
                                             cudaFuncAttributeMaxDynamicSharedMemorySize, Cfg<BN, FAM, CG>::SMEM);
        if (e != cudaSuccess) return dbl::cuda_check(e, "conv: set smem attribute");
        attr_set[dev] = true;
    }
    return DBL_OK;
}

// CTA pairs of conv_igemm_kernel<BN, FAM, 2> that fit on the device at once
// (cached per device); at most half the SMs and kMaxGrid / 2.
template <int BN, int FAM>
int resident_pairs()
{
    static int cached[64] = {0};
    int dev = -1;
    if (cudaGetDevice(&dev) != cudaSuccess) {
        (void)cudaGetLastError();
        dev = -1;
    }
    if (dev >= 0 && dev < 64 && cached[dev] > 0) return cached[dev];
    bool queried = false;  // only a plan the device itself answered for is cached
    int pairs = std::min(dbl::sm_count() / 2, kMaxGrid / 2);
    if (set_igemm_smem<BN, FAM, 2>() == DBL_OK) {
        cudaLaunchConfig_t cfg = {};
        cudaLaunchAttribute at[1];
        at[0].id = cudaLaunchAttributeClusterDimension;
        at[0].val.clusterDim.x = 2;
        at[0].val.clusterDim.y = 1;
        at[0].val.clusterDim.z = 1;
        cfg.gridDim = dim3(2 * pairs);
        cfg.blockDim = dim3(Cfg<BN, FAM, 2>::THREADS);
        cfg.dynamicSmemBytes = Cfg<BN, FAM, 2>::SMEM;
        cfg.attrs = at;
        cfg.numAttrs = 1;
        int n = 0;
        if (cudaOccupancyMaxActiveClusters(&n, conv_igemm_kernel<BN, FAM, 2>, &cfg) == cudaSuccess && n > 0)
        {
            pairs = std::min(pairs, n);
            queried = true;
        } else {
            (void)cudaGetLastError();
        }
    }
    if (pairs < 1) pairs = 1;
    if (queried && dev >= 0 && dev < 64) cached[dev] = pairs;
    return pairs;
}

// Persistent grid of a conv_igemm_kernel plan: one CTA per SM, or one CTA pair
// per two SMs, never more CTAs (pairs) than tiles.
int win_grid(const Plan& pl);

int plan_grid(const Plan& pl)
{
    if (pl.win) return win_grid(pl);
    if (pl.cg == 1) return grid_size(pl.p.total_tiles);
    const bool wg = pl.mode == kWgrad || pl.mode == kWgradC8;
    int pairs = pl.BN == 256 ? (wg ? resident_pairs<256, kFamWgrad>() : resident_pairs<256, kFamFwd>())
                             : (wg ? resident_pairs<128, kFamWgrad>() : resident_pairs<128, kFamFwd>());
    if (pairs > pl.p.total_tiles) pairs = pl.p.total_tiles;
    return 2 * std::max(pairs, 1);
}

// Launch attributes of a convolution kernel: a cluster of two for CTA pairs, and, with
// DBL_CONV_PDL=1 in the environment (read once per process), programmatic stream
// serialization, so that the kernel's set-up (barriers, TMEM, descriptor prefetch) overlaps the
// end of the kernel before it (its memory accesses wait in grid_dependency_wait).  Measured on
// GB300: one worker's 224 px step 1.2% faster with it; two workers' iteration on two streams
// 1.1% slower, because CTAs launched early wait on SMs the other stream's kernels need.  Off by
// default.
std::atomic<int> g_conv_pdl_override{-1};  // dbl_set_conv_pdl: -1 = the environment's choice
std::atomic<int> g_conv_stall_next{0};     // dbl_conv_test_stall_next: arms one implicit-GEMM launch

bool conv_pdl()
{
    static const bool env_on = [] {
        const char* e = getenv("DBL_CONV_PDL");
        return e && e[0] == '1';
    }();
    const int o = g_conv_pdl_override.load(std::memory_order_relaxed);
    return o < 0 ? env_on : o != 0;
}

int conv_attrs(int cg, cudaLaunchAttribute (&at)[2])
{
    int n = 0;
    if (cg == 2) {
        at[n].id = cudaLaunchAttributeClusterDimension;
        at[n].val.clusterDim.x = 2;
        at[n].val.clusterDim.y = 1;
        at[n].val.clusterDim.z = 1;
        ++n;
    }
    if (conv_pdl()) {
        at[n].id = cudaLaunchAttributeProgrammaticStreamSerialization;
        at[n].val.programmaticStreamSerializationAllowed = 1;
        ++n;
    }
    return n;
}

template <int BN, int FAM, int CG>
int launch_cfg(const Plan& pl, const CUtensorMap& a, const CUtensorMap& b, const CUtensorMap& a2,
               const CUtensorMap& b2, int grid, cudaStream_t st)
{
    using Cf = Cfg<BN, FAM, CG>;
    int rc = set_igemm_smem<BN, FAM, CG>();
    if (rc) return rc;
    cudaLaunchConfig_t cfg = {};
    cudaLaunchAttribute at[2];
    cfg.gridDim = dim3(grid);
    cfg.blockDim = dim3(Cf::THREADS);
    cfg.dynamicSmemBytes = Cf::SMEM;
    cfg.stream = st;
    cfg.attrs = at;
    cfg.numAttrs = conv_attrs(CG, at);
    ConvParams prm = pl.p;
    if (g_conv_stall_next.exchange(0)) prm.test_stall = 1;
    cudaError_t e = cudaLaunchKernelEx(&cfg, conv_igemm_kernel<BN, FAM, CG>, a, b, a2, b2, prm);
    if (e != cudaSuccess) {
        dbl::count_launch();
        return dbl::cuda_check(e, "conv_igemm launch");
    }
    return dbl::launch_check("conv_igemm launch");
}

// a2, b2: the projection operands of a fused data gradient (unused otherwise).
int launch(const Plan& pl, const CUtensorMap& a, const CUtensorMap& b, const CUtensorMap& a2, const CUtensorMap& b2,
           int grid, cudaStream_t st)
{
    const bool wg = pl.mode == kWgrad || pl.mode == kWgradC8;
    if (pl.cg == 2) {
        if (pl.BN == 256) return wg ? launch_cfg<256, kFamWgrad, 2>(pl, a, b, a2, b2, grid, st)
                                    : launch_cfg<256, kFamFwd, 2>(pl, a, b, a2, b2, grid, st);
        if (pl.BN == 128) return wg ? launch_cfg<128, kFamWgrad, 2>(pl, a, b, a2, b2, grid, st)
                                    : launch_cfg<128, kFamFwd, 2>(pl, a, b, a2, b2, grid, st);
        return dbl::set_error(DBL_ERR_UNSUPPORTED, "conv: CTA pairs need 128 or 256 columns per tile");
    }
    if (wg) {
        if (pl.BN == 256) return launch_cfg<256, kFamWgrad, 1>(pl, a, b, a2, b2, grid, st);
        if (pl.BN == 128) return launch_cfg<128, kFamWgrad, 1>(pl, a, b, a2, b2, grid, st);
        return launch_cfg<64, kFamWgrad, 1>(pl, a, b, a2, b2, grid, st);
    }
    if (pl.BN == 256) return launch_cfg<256, kFamFwd, 1>(pl, a, b, a2, b2, grid, st);
    if (pl.BN == 128) return launch_cfg<128, kFamFwd, 1>(pl, a, b, a2, b2, grid, st);
    return launch_cfg<64, kFamFwd, 1>(pl, a, b, a2, b2, grid, st);
}

template <int BN, bool DG, bool RES, int CG>
int set_win_smem()
{
    static bool attr_set[64] = {false};
    int dev = 0;
    cudaGetDevice(&dev);
    if (dev >= 0 && dev < 64 && !attr_set[dev]) {
        cudaError_t e = cudaFuncSetAttribute(conv_win_kernel<BN, DG, RES, CG>,
                                             cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kWinSmemMax);
        if (e != cudaSuccess) return dbl::cuda_check(e, "conv: set smem attribute");
        attr_set[dev] = true;
    }
    return DBL_OK;
}

// CTA pairs of conv_win_kernel<BN, DG, RES, 2> that fit on the device at once with
// `smem` bytes each (one CTA per SM; cached per device), at most half the SMs.
template <int BN, bool DG, bool RES>
int resident_win_pairs(size_t smem)
{
    static int cached[64] = {0};
    int dev = -1;
    if (cudaGetDevice(&dev) != cudaSuccess) {
        (void)cudaGetLastError();
        dev = -1;
    }
    if (dev >= 0 && dev < 64 && cached[dev] > 0) return cached[dev];
    bool queried = false;  // only a plan the device itself answered for is cached
    int pairs = std::min(dbl::sm_count() / 2, kMaxGrid / 2);
    if (set_win_smem<BN, DG, RES, 2>() == DBL_OK) {
        cudaLaunchConfig_t cfg = {};
        cudaLaunchAttribute at[1];
        at[0].id = cudaLaunchAttributeClusterDimension;
        at[0].val.clusterDim.x = 2;
        at[0].val.clusterDim.y = 1;
        at[0].val.clusterDim.z = 1;
        cfg.gridDim = dim3(2 * pairs);
        cfg.blockDim = dim3(WinCfg<BN>::THREADS);
        cfg.dynamicSmemBytes = smem;
        cfg.attrs = at;
        cfg.numAttrs = 1;
        int n = 0;
        if (cudaOccupancyMaxActiveClusters(&n, conv_win_kernel<BN, DG, RES, 2>, &cfg) == cudaSuccess && n > 0)
        {
            pairs = std::min(pairs, n);
            queried = true;
        } else {
            (void)cudaGetLastError();
        }
    }
    if (pairs < 1) pairs = 1;
    if (queried && dev >= 0 && dev < 64) cached[dev] = pairs;
    return pairs;
}

// Grid of a window-kernel plan: one CTA per SM (never more than tiles), or one CTA
// pair per two SMs (never more pairs than pair units).
int win_grid(const Plan& pl)
{
    if (pl.cg == 1) return grid_size(pl.p.total_tiles);
    const bool dg = pl.mode == kDgrad;
    int pairs = pl.BN == 64 ? resident_win_pairs<64, false, true>(pl.smem)
                : dg        ? resident_win_pairs<128, true, false>(pl.smem)
                            : resident_win_pairs<128, false, false>(pl.smem);
    const int units = (pl.p.total_tiles + 1) / 2;
    if (pairs > units) pairs = units;
    return 2 * std::max(pairs, 1);
}

template <int BN, bool DG, bool RES, int CG>
int launch_win_cfg(const Plan& pl, const CUtensorMap& a, const CUtensorMap& b, int grid, cudaStream_t st)
{
    int rc = set_win_smem<BN, DG, RES, CG>();
    if (rc) return rc;
    cudaLaunchConfig_t cfg = {};
    cudaLaunchAttribute at[2];
    cfg.gridDim = dim3(grid);
    cfg.blockDim = dim3(WinCfg<BN>::THREADS);
    cfg.dynamicSmemBytes = pl.smem;
    cfg.stream = st;
    cfg.attrs = at;
    cfg.numAttrs = conv_attrs(CG, at);
    cudaError_t e = cudaLaunchKernelEx(&cfg, conv_win_kernel<BN, DG, RES, CG>, a, b, pl.p);
    if (e != cudaSuccess) {
        dbl::count_launch();
        return dbl::cuda_check(e, "conv_win launch");
    }
    return dbl::launch_check("conv_win launch");
}

int launch_win(const Plan& pl, const CUtensorMap& a, const CUtensorMap& b, int grid, cudaStream_t st)
{
    const bool dg = pl.mode == kDgrad;
    if (pl.cg == 2) {
        if (pl.BN == 128) return dg ? launch_win_cfg<128, true, false, 2>(pl, a, b, grid, st)
                                    : launch_win_cfg<128, false, false, 2>(pl, a, b, grid, st);
        if (pl.BN == 64 && pl.res && !dg) return launch_win_cfg<64, false, true, 2>(pl, a, b, grid, st);
        return dbl::set_error(DBL_ERR_UNSUPPORTED, "conv: no CTA-pair window kernel for this plan");
    }
    if (pl.BN == 128) return dg ? launch_win_cfg<128, true, false, 1>(pl, a, b, grid, st)
                                : launch_win_cfg<128, false, false, 1>(pl, a, b, grid, st);
    if (pl.res) return dg ? launch_win_cfg<64, true, true, 1>(pl, a, b, grid, st)
                          : launch_win_cfg<64, false, true, 1>(pl, a, b, grid, st);
    return dg ? launch_win_cfg<64, true, false, 1>(pl, a, b, grid, st)
              : launch_win_cfg<64, false, false, 1>(pl, a, b, grid, st);
}

template <int NACC>
int launch_wgwin(const Plan& pl, const CUtensorMap& a, const CUtensorMap& b, cudaStream_t st)
{
    static bool attr_set[64] = {false};
    int dev = 0;
    cudaGetDevice(&dev);
    if (dev >= 0 && dev < 64 && !attr_set[dev]) {
        cudaError_t e = cudaFuncSetAttribute(conv_wgwin_kernel<NACC>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             (int)kWinSmemMax);
        if (e != cudaSuccess) return dbl::cuda_check(e, "conv: set smem attribute");
        attr_set[dev] = true;
    }
    cudaLaunchConfig_t cfg = {};
    cudaLaunchAttribute at[2];
    cfg.gridDim = dim3(grid_size(pl.p.zdim));
    cfg.blockDim = dim3(kWinThreads);
    cfg.dynamicSmemBytes = pl.smem;
    cfg.stream = st;
    cfg.attrs = at;
    cfg.numAttrs = conv_attrs(1, at);
    cudaError_t e = cudaLaunchKernelEx(&cfg, conv_wgwin_kernel<NACC>, a, b, pl.p);
    if (e != cudaSuccess) {
        dbl::count_launch();
        return dbl::cuda_check(e, "conv_wgwin launch");
    }
    return dbl::launch_check("conv_wgwin launch");
}

// Tensor map of the window kernel's strip operand: one padded row (Wp pixels
// x 64 channels, starting at w = -1) of an NHWC tensor per copy.
int enc_win_rows(CUtensorMap* m, const void* base, int N, int H, int W, int C, int Wp)
{
    cuuint64_t dims[4] = {(cuuint64_t)C, (cuuint64_t)W, (cuuint64_t)H, (cuuint64_t)N};
    cuuint64_t str[3] = {(cuuint64_t)C * 2, (cuuint64_t)W * C * 2, (cuuint64_t)H * W * C * 2};
    cuuint32_t box[4] = {64, (cuuint32_t)Wp, 1, 1};
    return enc_tiled(m, base, 4, dims, str, box, true);
}

// Rows of one tile of the forward family (see Cfg).
int fwd_tile_rows(int BN) { return BN <= 128 ? 256 : 128; }

// Forward pass.  nparts == nullptr: the channel sums are reduced into ch_sum/ch_sumsq
// (NULL: no statistics).  nparts != nullptr: the per-CTA partials are left in ws
// ([*nparts][2][k]) for the BatchNorm finalize to reduce (dbl_bn_relu_fused_parts).
int conv_fwd_impl(const dbl_conv_shape* s, const void* x, const void* w, void* y, float* ch_sum, float* ch_sumsq,
                  void* ws, size_t ws_bytes, int32_t* nparts, void* stream, const char* who)
{
    using namespace dbl;
    Plan pl;
    int rc = make_plan(s, DBL_PASS_FWD, pl);
    if (rc) return rc;
    if (!x || !w || !y || !aligned16(x) || !aligned16(w) || !aligned16(y))
        return set_error(DBL_ERR_INVALID, "%s: null or misaligned tensor", who);
    if ((ch_sum == nullptr) != (ch_sumsq == nullptr))
        return set_error(DBL_ERR_INVALID, "%s: ch_sum and ch_sumsq go together", who);
    const bool stats = ch_sum != nullptr || nparts != nullptr;
    if (stats && (!ws || ws_bytes < plan_ws(pl)))
        return set_error(DBL_ERR_WORKSPACE, "%s: workspace %zu < %zu bytes", who, ws_bytes, plan_ws(pl));
    CUtensorMap ta, tb;
    const Geom g = geom(s);
    if (pl.win) {
        if ((rc = enc_win_rows(&ta, x, s->n, s->h, s->w, s->c, pl.p.win_Wp))) return rc;
        const int64_t rsc = (int64_t)s->r * s->s * s->c;
        cuuint64_t dims[2] = {(cuuint64_t)rsc, (cuuint64_t)s->k};
        cuuint64_t str[1] = {(cuuint64_t)rsc * 2};
        cuuint32_t box[2] = {64, (cuuint32_t)(pl.BN / pl.cg)};  // a CTA pair stages half the columns each
        if ((rc = enc_tiled(&tb, w, 2, dims, str, box, true))) return rc;
    } else if (pl.mode == kFwdC8) {
        if ((rc = enc_im2col(&ta, x, s->n, s->h, s->w, 8, -g.ph, g.ph - (s->r - 1), -g.pw, g.pw - (s->s - 1), g.sh,
                             g.sw, 8, fwd_tile_rows(pl.BN), false)))
            return rc;
        const int64_t rsc = (int64_t)s->r * s->s * 8;
        cuuint64_t dims[2] = {(cuuint64_t)rsc, (cuuint64_t)s->k};
        cuuint64_t str[1] = {(cuuint64_t)rsc * 2};
        cuuint32_t box[2] = {8, (cuuint32_t)pl.BN};
        if ((rc = enc_tiled(&tb, w, 2, dims, str, box, false))) return rc;
    } else {
        if ((rc = enc_im2col(&ta, x, s->n, s->h, s->w, s->c, -g.ph, g.ph - (s->r - 1), -g.pw, g.pw - (s->s - 1), g.sh,
                             g.sw, 64, fwd_tile_rows(pl.BN), true)))
            return rc;
        const int64_t rsc = (int64_t)s->r * s->s * s->c;
        cuuint64_t dims[2] = {(cuuint64_t)rsc, (cuuint64_t)s->k};
        cuuint64_t str[1] = {(cuuint64_t)rsc * 2};
        cuuint32_t box[2] = {64, (cuuint32_t)(pl.BN / pl.cg)};
        if ((rc = enc_tiled(&tb, w, 2, dims, str, box, true))) return rc;
    }
    pl.p.out = y;
    pl.p.st32 = (reinterpret_cast<uintptr_t>(y) % 32 == 0) && (pl.p.ldo * (int64_t)sizeof(act_t)) % 32 == 0;
    pl.p.stats = stats ? static_cast<float*>(ws) : nullptr;
    const int grid = plan_grid(pl);
    cudaStream_t st = as_stream(stream);
    if ((rc = pl.win ? launch_win(pl, ta, tb, grid, st) : launch(pl, ta, tb, ta, tb, grid, st))) return rc;
    if (nparts) {
        *nparts = grid;
    } else if (stats) {
        stats_reduce_kernel<<<(s->k + kPartialsChannels - 1) / kPartialsChannels, kPartialsThreads, 0, st>>>(pl.p.stats, grid, s->k, ch_sum, ch_sumsq);
        if ((rc = launch_check("conv stats reduce"))) return rc;
    }
    return DBL_OK;
}


// Data gradient, optionally with the projection shortcut of a ResNet block fused in:
// k2 > 0 adds dgrad of a 1x1 stride-2 pad-0 convolution of the same input (dy2:
// [n, h/2, w/2, k2], w2: [k2][c]) to phase (0,0), the only phase it reaches.
int conv_dgrad_impl(const dbl_conv_shape* s, const void* dy, const void* w, int k2, const void* dy2, const void* w2,
                    void* dx, void* stream, const char* who)
{
    using namespace dbl;
    Plan pl;
    int rc = make_plan(s, DBL_PASS_DGRAD, pl);
    if (rc) return rc;
    if (!dy || !w || !dx || !aligned16(dy) || !aligned16(w) || !aligned16(dx))
        return set_error(DBL_ERR_INVALID, "%s: null or misaligned tensor", who);
    const int P = out_dim(s->h, s->r, s->stride, s->pad), Q = out_dim(s->w, s->s, s->stride, s->pad);
    CUtensorMap ta, tb, ta2, tb2;
    if (pl.win) {
        if ((rc = enc_win_rows(&ta, dy, s->n, P, Q, s->k, pl.p.win_Wp))) return rc;
    } else {
        // im2col over dy [n, P, Q, k]: origins cover the dx grid (stride 1) or one phase grid (stride 2)
        int lower = 0, upper = 0;
        if (s->stride == 1) {
            lower = -(s->r - 1 - s->pad);
            upper = (s->h - 1 + lower) - (P - 1);  // origin range [lower, H-1+lower] against dy's extent P
        }
        if ((rc = enc_im2col(&ta, dy, s->n, P, Q, s->k, lower, upper, lower, upper, 1, 1, 64, fwd_tile_rows(pl.BN),
                             true)))
            return rc;
    }
    // w viewed as [k][r*s][c]: inner c, then tap, then k
    cuuint64_t dims[3] = {(cuuint64_t)s->c, (cuuint64_t)s->r * s->s, (cuuint64_t)s->k};
    cuuint64_t str[2] = {(cuuint64_t)s->c * 2, (cuuint64_t)s->r * s->s * s->c * 2};
    cuuint32_t box[3] = {64, 1, 64};
    if ((rc = enc_tiled(&tb, w, 3, dims, str, box, true))) return rc;
    ta2 = ta;
    tb2 = tb;
    if (k2 > 0) {
        if (pl.win || pl.p.phase_div != 2)
            return set_error(DBL_ERR_UNSUPPORTED, "%s: the projection needs the stride-2 phase path", who);
        // dy2 [n, h/2, w/2, k2] = the phase grid's rows, as [n*P*Q][k2]
        cuuint64_t d2[2] = {(cuuint64_t)k2, (cuuint64_t)s->n * pl.p.gP * pl.p.gQ};
        cuuint64_t s2[1] = {(cuuint64_t)k2 * 2};
        cuuint32_t bx2[2] = {64, (cuuint32_t)fwd_tile_rows(pl.BN)};
        if ((rc = enc_tiled(&ta2, dy2, 2, d2, s2, bx2, true))) return rc;
        // w2 [k2][c] viewed as [k2][1][c], loaded like one tap of w
        cuuint64_t d3[3] = {(cuuint64_t)s->c, 1, (cuuint64_t)k2};
        cuuint64_t s3[2] = {(cuuint64_t)s->c * 2, (cuuint64_t)s->c * 2};
        if ((rc = enc_tiled(&tb2, w2, 3, d3, s3, box, true))) return rc;
        pl.p.proj_kb = k2 / 64;
    }
    pl.p.out = dx;
    pl.p.st32 = (reinterpret_cast<uintptr_t>(dx) % 32 == 0) && (pl.p.ldo * (int64_t)sizeof(act_t)) % 32 == 0;
    const int grid = plan_grid(pl);
    return pl.win ? launch_win(pl, ta, tb, grid, as_stream(stream))
                  : launch(pl, ta, tb, ta2, tb2, grid, as_stream(stream));
}

}  // namespace

extern "C" {

size_t dbl_conv_workspace_bytes(const dbl_conv_shape* shape, int pass)
{
    Plan pl;
    if (pass < 0 || pass > 2 || make_plan(shape, pass, pl) != DBL_OK) return 0;
    return plan_ws(pl);
}

int dbl_conv_plan(const dbl_conv_shape* s, int pass, dbl_conv_plan_info* info)
{
    using namespace dbl;
    if (!info || pass < 0 || pass > 2) return set_error(DBL_ERR_INVALID, "conv_plan: bad arguments");
    Plan pl;
    int rc = make_plan(s, pass, pl);
    if (rc) return rc;
    const bool wgwin = pl.win && pass == DBL_PASS_WGRAD;
    info->kernel = wgwin ? DBL_KERNEL_WINDOW_WGRAD : pl.win ? DBL_KERNEL_WINDOW : DBL_KERNEL_IGEMM;
    info->tile_cols = wgwin ? s->k : pl.BN;
    info->ctas_per_mma = pl.cg;
    info->tiles = pl.p.total_tiles;
    info->zdim = pl.p.zdim;
    info->grid = wgwin ? grid_size(pl.p.zdim) : plan_grid(pl);
    info->smem_bytes = pl.win ? (int64_t)pl.smem : 0;
    return DBL_OK;
}

int dbl_conv_fwd(const dbl_conv_shape* s, const void* x, const void* w, void* y, float* ch_sum, float* ch_sumsq,
                 void* ws, size_t ws_bytes, void* stream)
{
    return conv_fwd_impl(s, x, w, y, ch_sum, ch_sumsq, ws, ws_bytes, nullptr, stream, "conv_fwd");
}

size_t dbl_conv_stats_parts_bytes(const dbl_conv_shape* shape)
{
    Plan pl;
    if (make_plan(shape, DBL_PASS_FWD, pl) != DBL_OK) return 0;
    return (size_t)kMaxGrid * 2 * shape->k * sizeof(float);
}

int dbl_conv_fwd_parts(const dbl_conv_shape* s, const void* x, const void* w, void* y, float* parts,
                       size_t parts_bytes, int32_t* nparts, void* stream)
{
    using dbl::set_error;
    if (!parts || !nparts) return set_error(DBL_ERR_INVALID, "conv_fwd_parts: null partials or count");
    return conv_fwd_impl(s, x, w, y, nullptr, nullptr, parts, parts_bytes, nparts, stream, "conv_fwd_parts");
}

int dbl_conv_dgrad(const dbl_conv_shape* s, const void* dy, const void* w, void* dx, void* ws, size_t ws_bytes,
                   void* stream)
{
    (void)ws;
    (void)ws_bytes;
    return conv_dgrad_impl(s, dy, w, 0, nullptr, nullptr, dx, stream, "conv_dgrad");
}

int dbl_conv_dgrad_proj(const dbl_conv_shape* s, const void* dy, const void* w, int32_t k2, const void* dy2,
                        const void* w2, void* dx, void* ws, size_t ws_bytes, void* stream)
{
    (void)ws;
    (void)ws_bytes;
    using dbl::set_error;
    if (!s) return set_error(DBL_ERR_INVALID, "conv_dgrad_proj: null shape");
    if (s->stride != 2 || (s->stride_w && s->stride_w != 2))
        return set_error(DBL_ERR_UNSUPPORTED, "conv_dgrad_proj: the main convolution must have stride 2");
    if (k2 <= 0 || k2 % 64 || k2 > kMaxNcols)
        return set_error(DBL_ERR_UNSUPPORTED, "conv_dgrad_proj: projection channels must be a multiple of 64, <= %d",
                         kMaxNcols);
    if (!dy2 || !w2 || !dbl::aligned16(dy2) || !dbl::aligned16(w2))
        return set_error(DBL_ERR_INVALID, "conv_dgrad_proj: null or misaligned projection tensor");
    return conv_dgrad_impl(s, dy, w, k2, dy2, w2, dx, stream, "conv_dgrad_proj");
}

int dbl_conv_wgrad(const dbl_conv_shape* s, const void* x, const void* dy, float* dw, int accumulate, void* ws,
                   size_t ws_bytes, void* stream)
{
    using namespace dbl;
    Plan pl;
    int rc = make_plan(s, DBL_PASS_WGRAD, pl);
    if (rc) return rc;
    if (!x || !dy || !dw || !aligned16(x) || !aligned16(dy) || !aligned16(dw))
        return set_error(DBL_ERR_INVALID, "conv_wgrad: null or misaligned tensor");
    if (plan_ws(pl) && (!ws || ws_bytes < plan_ws(pl)))
        return set_error(DBL_ERR_WORKSPACE, "conv_wgrad: workspace %zu < %zu bytes", ws_bytes, plan_ws(pl));
    const Geom g = geom(s);
    const int P = out_dim(s->h, s->r, g.sh, g.ph), Q = out_dim(s->w, s->s, g.sw, g.pw);
    CUtensorMap ta, tb;
    cudaStream_t st = as_stream(stream);
    const bool sliced = pl.p.zdim > 1;
    if (pl.win) {
        if ((rc = enc_win_rows(&ta, x, s->n, s->h, s->w, s->c, pl.p.win_Wp))) return rc;
        if ((rc = enc_win_rows(&tb, dy, s->n, P, Q, s->k, pl.p.win_Wp))) return rc;
        pl.p.out = sliced ? ws : static_cast<void*>(dw);
        pl.p.wg_accumulate = accumulate;
        const int nacc = (pl.p.win_R * pl.p.win_S + 1) / 2;
        if ((rc = nacc == 5 ? launch_wgwin<5>(pl, ta, tb, st) : launch_wgwin<2>(pl, ta, tb, st))) return rc;
    } else {
    const bool c8 = pl.mode == kWgradC8;
    if ((rc = enc_im2col(&ta, x, s->n, s->h, s->w, s->c, -g.ph, g.ph - (s->r - 1), -g.pw, g.pw - (s->s - 1), g.sh, g.sw,
                         c8 ? 8 : 64, 128, !c8)))
        return rc;
    cuuint64_t dims[2] = {(cuuint64_t)s->k, (cuuint64_t)s->n * P * Q};
    cuuint64_t str[1] = {(cuuint64_t)s->k * 2};
    cuuint32_t box[2] = {64, 128};
    if ((rc = enc_tiled(&tb, dy, 2, dims, str, box, true))) return rc;
    pl.p.out = sliced ? ws : static_cast<void*>(dw);
    pl.p.wg_accumulate = accumulate;
    if ((rc = launch(pl, ta, tb, ta, tb, plan_grid(pl), st))) return rc;
    }
    if (!sliced) return DBL_OK;
    const int64_t n = (int64_t)pl.p.M * s->k;
    const int lanes = pl.p.zdim > 8 ? 8 : 1;
    int64_t blocks = (n / 4 + 256 / lanes - 1) / (256 / lanes);
    const int64_t cap = (int64_t)sm_count() * 8;
    if (blocks > cap) blocks = cap;
    if (blocks < 1) blocks = 1;
    if (lanes == 8)
        wgrad_reduce_kernel<8><<<(int)blocks, 256, 0, st>>>(static_cast<const float*>(ws), pl.p.zdim, n, dw, accumulate);
    else
        wgrad_reduce_kernel<1><<<(int)blocks, 256, 0, st>>>(static_cast<const float*>(ws), pl.p.zdim, n, dw, accumulate);
    return launch_check("conv wgrad reduce");
}

int dbl_device_status(int32_t* status)
{
    using namespace dbl;
    if (!status) return set_error(DBL_ERR_INVALID, "device_status: null");
    int rc = cuda_check(cudaDeviceSynchronize(), "device_status sync");
    if (rc) return rc;
    int v = 0, zero = 0;
    if ((rc = cuda_check(cudaMemcpyFromSymbol(&v, g_conv_status, sizeof(int)), "device_status read"))) return rc;
    if ((rc = cuda_check(cudaMemcpyToSymbol(g_conv_status, &zero, sizeof(int)), "device_status clear"))) return rc;
    *status = v;
    return DBL_OK;
}

}  // extern "C"

extern "C" int dbl_conv_test_stall_next(void)
{
    g_conv_stall_next.store(1);
    return DBL_OK;
}

extern "C" int dbl_set_conv_pdl(int32_t mode)
{
    if (mode < -1 || mode > 1) return dbl::set_error(DBL_ERR_INVALID, "set_conv_pdl: mode must be -1, 0 or 1");
    g_conv_pdl_override.store(mode, std::memory_order_relaxed);
    return DBL_OK;
}
