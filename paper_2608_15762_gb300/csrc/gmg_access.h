// Access to a created GMG's device graph for the library's translation units
// other than the simulator's (private to the library, not part of the C ABI).
#pragma once

#include "gmg_layout.h"

namespace gsim {

// The device graph of g (defined in gmgsim_host.cu); nullptr for nullptr.
const DevGmg* gmg_device_graph(const gmg_t* g);

}  // namespace gsim
