// heddle_tiled.cuh -- expert tiling (§5.3 "Expert tiling"): the tables and
// the search that price a stage's devices as EP x ETP x EDP.

#pragma once

#include "heddle_internal.cuh"

namespace hd {

constexpr int kTileSlots = 20;  // tilings of 1, 2, 4, 8 devices: 1 + 3 + 6 + 10

// First slot of each degree 2^j; slot order within a degree is EDP exponent
// ascending, then ETP exponent ascending (EP takes the rest).
__host__ __device__ inline int tile_base(int j) { return j == 0 ? 0 : j == 1 ? 1 : j == 2 ? 4 : 10; }

// Byte layout of the tiled image, staged into shared memory by the search.
struct TiledLayout {
    int32_t L, NT;
    uint32_t offPt;     // int64 [NT][20][L+1]  prefix of per-layer ns per (type, tiling slot)
    uint32_t offSA;     // int64x2 [L+1]         prefix of (state bytes, activation bytes)
    uint32_t offES;     // int64 [L+1]           prefix of the experts' state bytes
    uint32_t offPB;     // int64 [L+1]           prefix of gradient bytes
    uint32_t offPE;     // int64 [L+1]           prefix of the experts' gradient bytes
    uint32_t offP2P;    // int64 [8][8][2]       P2P ns (from, to, same-node)
    uint32_t offMem;    // int64 [8]             memory per GPU
    uint32_t offInter;  // int64 [8]             slowest NIC of the type
    uint32_t offIntra;  // int64 [8]             intra-node bandwidth of the type
    uint32_t offMaxN;   // int32 [8]             largest node of the type
    uint32_t offCode;   // uint8 [8][20]         log2 EP | log2 ETP << 2 | log2 EDP << 4,
                        //                       bit 7 set when the tiling is allowed
    uint32_t bytes;
};

inline TiledLayout make_tiled_layout(int L, int NT) {
    TiledLayout y{};
    y.L = L;
    y.NT = NT;
    uint32_t o = 0;
    y.offPt = o;    o = align16(o + 8u * NT * kTileSlots * (L + 1));
    y.offSA = o;    o = align16(o + 16u * (L + 1));
    y.offES = o;    o = align16(o + 8u * (L + 1));
    y.offPB = o;    o = align16(o + 8u * (L + 1));
    y.offPE = o;    o = align16(o + 8u * (L + 1));
    y.offP2P = o;   o = align16(o + 8u * 8 * 8 * 2);
    y.offMem = o;   o = align16(o + 8u * 8);
    y.offInter = o; o = align16(o + 8u * 8);
    y.offIntra = o; o = align16(o + 8u * 8);
    y.offMaxN = o;  o = align16(o + 4u * 8);
    y.offCode = o;  o = align16(o + 8u * kTileSlots);
    y.bytes = o;
    return y;
}

// Largest tiled image the search stages into shared memory.
constexpr uint32_t kTiledImageLimit = 160u * 1024u;

struct TiledTableArgs {
    TiledLayout tl;
    Layout lay;                  // the main image it reads node statistics, P2P and bytes from
    const unsigned char* img;    // main image (device)
    const heddle_gpu_type* types;
    const heddle_layer* layers;
    const int64_t* expert_state;  // [L]
    const int64_t* expert_param;  // [L]
    unsigned char* timg;         // tiled image (device, out)
    uint32_t* flags;             // kTab* bits
};

cudaError_t launch_tiled_tables(const TiledTableArgs& a, cudaStream_t st);

struct TiledArgs {
    TiledLayout tl;
    const unsigned char* timg;
    uint8_t* tiling;   // nullable: chosen tiling per stage, plane s at tiling[s * tstride + c]
    int64_t tstride;
};

// Screen launch (and, with `mid`, the event after it) of the pricing path.
cudaError_t launch_screen(const PriceArgs& a, int num_sms, cudaStream_t st, cudaEvent_t mid, int64_t* launches);

// Tiled PartitionLayers + Evaluate over the screen's worklist.
cudaError_t launch_tiled_search(const PriceArgs& a, const TiledArgs& t, int num_sms, cudaStream_t st);

}  // namespace hd
